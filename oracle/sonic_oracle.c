/*
 * Double-precision CPU oracle for the SONIC Nexus-KV attention path.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, plain statement of what
 * the CUDA library computes.  Only the tests, the smoke entry point and the
 * CPU-baseline leg of the benchmark may load it; the library itself never
 * calls it and shares no code, header or constant with it.
 *
 * Everything works on host memory, in plain loops, in double precision,
 * following the paper (SONIC, arXiv 2601.21927) section by section:
 *
 *   orc_visible       -- the hierarchical visibility mask of Sec. 3.2
 *                        (Eq. 3 causal rule, Eq. 4 historical body removal,
 *                        Eq. 5 bidirectional Nexus visibility), evaluated for
 *                        one (query p, key q) pair.
 *   orc_retain        -- the KV retention rule: after the mask, only the
 *                        system prompt, the Nexus tokens and the current
 *                        query stay (Sec. 1, Fig. 2 caption, Sec. 3.2 body
 *                        removal, App. C effective context).
 *   orc_compact_copy  -- the byte copy of the retained rows, in original
 *                        order.
 *   orc_attn_masked   -- softmax attention under the additive mask M of
 *                        Sec. 3.2 (M = 0 visible, -inf hidden), grouped-query
 *                        head mapping h -> h / (Hq/Hkv).
 *   orc_decode        -- one generation step over the retained cache
 *                        (App. C: the effective context is I_sys, the Nexus
 *                        state and Q_n); every retained row is visible.
 *
 * Readings where the paper is silent (documented with the design notes):
 *   - A pair with exactly one Nexus token follows the global causal rule
 *     ("no token can attend to future text tokens", Sec. 3.2).
 *   - A segment with zero Nexus tokens hides its body from every later
 *     position, as if max(N_i) were the segment's last token (Sec. 3.2,
 *     Sec. 4.2 allows reducing K for short segments).
 *   - Nexus-to-Nexus visibility is total across all segments (Eq. 5,
 *     "fully connected memory graph"); the alternative reading, where a
 *     Nexus token sees only Nexus tokens of its own and earlier segments
 *     (Nexus kept across a session, Sec. 6.4), is nexus_mode = 1.
 *   - The softmax scale is 1/sqrt(D) unless the caller passes another.
 *   - A query row with no visible key outputs zeros and lse = -inf.
 *
 * Parity pins for every function live in tests/test_oracle_pins.py.
 */
#include <math.h>
#include <stdint.h>
#include <stddef.h>
#include <string.h>

#define ORC_SYS 0
#define ORC_BODY 1
#define ORC_NEXUS 2
#define ORC_CURR 3

#define ORC_NEXUS_FULL 0
#define ORC_NEXUS_CAUSAL_SEGMENTS 1

/*
 * Sec. 3.2: is key q visible to query p?  p, q are positions in the
 * augmented sequence S_aug (Eq. 1); role/seg are the per-token role and
 * segment number (0 = system prompt, 1..h = history segment m_i,
 * h+1 = current query).
 */
int orc_visible(int64_t p, int64_t q, const uint8_t *role, const int32_t *seg,
                int nexus_mode)
{
    uint8_t rp = role[p], rq = role[q];
    if (rq == ORC_BODY) {
        /* Eq. 4: body tokens B_i are hidden from every position after
         * max(N_i).  Segments are contiguous [B_i, N_i], so a position
         * p >= q that has not passed max(N_i) lies in segment i itself;
         * positions of other segments never see B_i.  Eq. 3 still applies
         * inside the segment (q <= p). */
        return seg[q] == seg[p] && q <= p;
    }
    if (rp == ORC_NEXUS && rq == ORC_NEXUS) {
        /* Eq. 5 and the within-segment bidirectional rule. */
        if (nexus_mode == ORC_NEXUS_FULL)
            return 1;
        return seg[q] <= seg[p];
    }
    /* Eq. 3, applied globally: no token attends to a future text token. */
    return q <= p;
}

/*
 * Retention: keep[t] = (role[t] != BODY).  For each sequence b
 * (rows k_start[b] .. k_start[b]+k_len[b]-1 of the packed token axis):
 *   ret_len[b]  = number of kept rows,
 *   offsets[b]  = sum over b' < b of (ret_len[b'] + reserve[b']),
 *   src_idx[offsets[b] + j] = packed index of the j-th kept row, in order.
 * Rows offsets[b]+ret_len[b] .. offsets[b+1]-1 are the caller's reserve
 * and are left untouched (src_idx not written there).
 * Returns offsets[B], the total number of output rows.
 */
int64_t orc_retain(int32_t B, const int32_t *k_start, const int32_t *k_len,
                   const uint8_t *role, const int32_t *reserve,
                   int32_t *offsets, int32_t *ret_len, int32_t *src_idx)
{
    int64_t off = 0;
    for (int32_t b = 0; b < B; ++b) {
        offsets[b] = (int32_t)off;
        int32_t n = 0;
        for (int32_t t = 0; t < k_len[b]; ++t) {
            int32_t row = k_start[b] + t;
            if (role[row] != ORC_BODY) {
                if (src_idx)
                    src_idx[off + n] = row;
                ++n;
            }
        }
        if (ret_len)
            ret_len[b] = n;
        off += n + (reserve ? reserve[b] : 0);
    }
    offsets[B] = (int32_t)off;
    return off;
}

/*
 * Copy the retained rows of every layer: for each layer l and each
 * sequence b, output row offsets[b]+j of layer l receives the bytes of
 * input row src_idx[offsets[b]+j] of layer l.  row_bytes is the size of
 * one token row (all KV heads); layer strides are in bytes.
 */
void orc_compact_copy(int32_t B, int32_t n_layers, const uint8_t *src,
                      int64_t src_layer_bytes, const int32_t *offsets,
                      const int32_t *ret_len, const int32_t *src_idx,
                      int64_t row_bytes, uint8_t *dst, int64_t dst_layer_bytes)
{
    for (int32_t l = 0; l < n_layers; ++l)
        for (int32_t b = 0; b < B; ++b)
            for (int32_t j = 0; j < ret_len[b]; ++j) {
                int64_t o = (int64_t)offsets[b] + j;
                memcpy(dst + l * dst_layer_bytes + o * row_bytes,
                       src + l * src_layer_bytes + (int64_t)src_idx[o] * row_bytes,
                       (size_t)row_bytes);
            }
}

/*
 * Masked softmax attention for selected query rows of ONE sequence.
 *   K, V : [L][Hkv][D]   (the sequence's key/value rows, S_aug order)
 *   Q    : [n_rows][Hq][D]
 *   rows : [n_rows]      position in S_aug of each query row
 *   O    : [n_rows][Hq][D]
 *   lse  : [n_rows][Hq]  natural-log log-sum-exp of the scaled, visible
 *                        scores (nullable)
 * For query head h the key/value head is h / (Hq / Hkv).
 * s_q = scale * <Q[p,h], K[q,h/G]>, M_{p,q} = 0 if orc_visible else -inf,
 * O[p,h] = sum_q softmax(s + M)_q V[q,h/G].
 */
void orc_attn_masked(int64_t L, int32_t Hq, int32_t Hkv, int32_t D,
                     const double *Q, const double *K, const double *V,
                     const uint8_t *role, const int32_t *seg,
                     const int64_t *rows, int64_t n_rows, double scale,
                     int nexus_mode, double *s_buf, double *O, double *lse)
{
    /* s_buf: caller-provided scratch of L doubles. */
    int32_t G = Hq / Hkv;
    for (int64_t i = 0; i < n_rows; ++i) {
        int64_t p = rows[i];
        for (int32_t h = 0; h < Hq; ++h) {
            int32_t hk = h / G;
            const double *qv = Q + (i * Hq + h) * (int64_t)D;
            double m = -INFINITY;
            for (int64_t q = 0; q < L; ++q) {
                if (!orc_visible(p, q, role, seg, nexus_mode)) {
                    s_buf[q] = -INFINITY;
                    continue;
                }
                const double *kv = K + (q * Hkv + hk) * (int64_t)D;
                double s = 0.0;
                for (int32_t d = 0; d < D; ++d)
                    s += qv[d] * kv[d];
                s *= scale;
                s_buf[q] = s;
                if (s > m)
                    m = s;
            }
            double *o = O + (i * Hq + h) * (int64_t)D;
            for (int32_t d = 0; d < D; ++d)
                o[d] = 0.0;
            if (m == -INFINITY) {
                if (lse)
                    lse[i * Hq + h] = -INFINITY;
                continue;
            }
            double denom = 0.0;
            for (int64_t q = 0; q < L; ++q) {
                if (s_buf[q] == -INFINITY)
                    continue;
                double w = exp(s_buf[q] - m);
                denom += w;
                const double *vv = V + (q * Hkv + hk) * (int64_t)D;
                for (int32_t d = 0; d < D; ++d)
                    o[d] += w * vv[d];
            }
            for (int32_t d = 0; d < D; ++d)
                o[d] /= denom;
            if (lse)
                lse[i * Hq + h] = m + log(denom);
        }
    }
}

/*
 * One decode step of one sequence over its retained cache (App. C):
 *   q : [Hq][D], K, V : [n][Hkv][D] (the n retained rows, the new token's
 *   own row included), O : [Hq][D], lse : [Hq] (nullable).
 * Every retained row is visible to the new token.
 */
void orc_decode(int64_t n, int32_t Hq, int32_t Hkv, int32_t D, const double *q,
                const double *K, const double *V, double scale, double *s_buf,
                double *O, double *lse)
{
    int32_t G = Hq / Hkv;
    for (int32_t h = 0; h < Hq; ++h) {
        int32_t hk = h / G;
        const double *qv = q + (int64_t)h * D;
        double m = -INFINITY;
        for (int64_t t = 0; t < n; ++t) {
            const double *kv = K + (t * Hkv + hk) * (int64_t)D;
            double s = 0.0;
            for (int32_t d = 0; d < D; ++d)
                s += qv[d] * kv[d];
            s *= scale;
            s_buf[t] = s;
            if (s > m)
                m = s;
        }
        double *o = O + (int64_t)h * D;
        for (int32_t d = 0; d < D; ++d)
            o[d] = 0.0;
        if (n == 0) {
            if (lse)
                lse[h] = -INFINITY;
            continue;
        }
        double denom = 0.0;
        for (int64_t t = 0; t < n; ++t) {
            double w = exp(s_buf[t] - m);
            denom += w;
            const double *vv = V + (t * Hkv + hk) * (int64_t)D;
            for (int32_t d = 0; d < D; ++d)
                o[d] += w * vv[d];
        }
        for (int32_t d = 0; d < D; ++d)
            o[d] /= denom;
        if (lse)
            lse[h] = m + log(denom);
    }
}

/*
 * Attention mass on Nexus keys: the per-row, per-head quantity behind
 * A_nexus of the Nexus attention regularisation (Sec. 4.1, Eq. 9, "the
 * average attention weight assigned to Nexus tokens by the current query").
 * For each selected query row p and query head h, with the softmax of
 * orc_attn_masked (scores s_q over the keys visible to p under the Sec. 3.2
 * rule):
 *   mass[p,h] = sum_{q visible, role[q] = NEXUS} e^{s_q}
 *             / sum_{q visible} e^{s_q},
 * 0 when p sees no key.  Same argument layout as orc_attn_masked; mass is
 * [n_rows][Hq].
 */
void orc_nexus_mass(int64_t L, int32_t Hq, int32_t Hkv, int32_t D,
                    const double *Q, const double *K, const uint8_t *role,
                    const int32_t *seg, const int64_t *rows, int64_t n_rows,
                    double scale, int nexus_mode, double *s_buf, double *mass)
{
    int32_t G = Hq / Hkv;
    for (int64_t i = 0; i < n_rows; ++i) {
        int64_t p = rows[i];
        for (int32_t h = 0; h < Hq; ++h) {
            int32_t hk = h / G;
            const double *qv = Q + (i * Hq + h) * (int64_t)D;
            double m = -INFINITY;
            for (int64_t q = 0; q < L; ++q) {
                if (!orc_visible(p, q, role, seg, nexus_mode)) {
                    s_buf[q] = -INFINITY;
                    continue;
                }
                const double *kv = K + (q * Hkv + hk) * (int64_t)D;
                double s = 0.0;
                for (int32_t d = 0; d < D; ++d)
                    s += qv[d] * kv[d];
                s *= scale;
                s_buf[q] = s;
                if (s > m)
                    m = s;
            }
            double all = 0.0, nexus = 0.0;
            for (int64_t q = 0; q < L; ++q) {
                if (s_buf[q] == -INFINITY)
                    continue;
                double w = exp(s_buf[q] - m);
                all += w;
                if (role[q] == ORC_NEXUS)
                    nexus += w;
            }
            mass[i * Hq + h] = all > 0.0 ? nexus / all : 0.0;
        }
    }
}

/*
 * The same mass for one decode step (App. C): the new token's query q
 * [Hq][D] sees every one of the n retained rows K [n][Hkv][D], whose roles
 * are role[n]; mass is [Hq], 0 when n = 0.
 */
void orc_decode_nexus_mass(int64_t n, int32_t Hq, int32_t Hkv, int32_t D,
                           const double *q, const double *K, const uint8_t *role,
                           double scale, double *s_buf, double *mass)
{
    int32_t G = Hq / Hkv;
    for (int32_t h = 0; h < Hq; ++h) {
        int32_t hk = h / G;
        const double *qv = q + (int64_t)h * D;
        double m = -INFINITY;
        for (int64_t t = 0; t < n; ++t) {
            const double *kv = K + (t * Hkv + hk) * (int64_t)D;
            double s = 0.0;
            for (int32_t d = 0; d < D; ++d)
                s += qv[d] * kv[d];
            s *= scale;
            s_buf[t] = s;
            if (s > m)
                m = s;
        }
        double all = 0.0, nexus = 0.0;
        for (int64_t t = 0; t < n; ++t) {
            double w = exp(s_buf[t] - m);
            all += w;
            if (role[t] == ORC_NEXUS)
                nexus += w;
        }
        mass[h] = all > 0.0 ? nexus / all : 0.0;
    }
}

/*
 * Role-routed linear map (Sec. 3.1, "Nexus Insertion and Representation":
 * Nexus tokens get dedicated projection matrices W_Q^N, W_K^N, W_V^N, W_O^N,
 * every other token the model's own):
 *   Y[t][n] = sum_k X[t][k] * Wsel(t)[n][k],
 *   Wsel(t) = W_nexus if role[t] is NEXUS, W otherwise.
 * X is [T][d_in]; W and W_nexus are [d_out][d_in] (the out x in layout of a
 * linear layer); Y is [T][d_out].
 */
void orc_routed_linear(int64_t T, int32_t d_in, int32_t d_out, const double *X,
                       const double *W, const double *W_nexus, const uint8_t *role,
                       double *Y)
{
    for (int64_t t = 0; t < T; ++t) {
        const double *w = role[t] == ORC_NEXUS ? W_nexus : W;
        const double *x = X + t * (int64_t)d_in;
        for (int32_t n = 0; n < d_out; ++n) {
            const double *wn = w + (int64_t)n * d_in;
            double acc = 0.0;
            for (int32_t k = 0; k < d_in; ++k)
                acc += x[k] * wn[k];
            Y[t * (int64_t)d_out + n] = acc;
        }
    }
}
