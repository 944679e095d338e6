// Masked prefill: flash-style attention under SONIC's hierarchical visibility
// mask (Sec. 3.2: Eq. 3 causal rule, Eq. 4 historical body removal, Eq. 5
// bidirectional Nexus visibility), on the sm_103a tensor cores.
//
// A work unit is two 128-row query tiles of one (layer, sequence): one query
// block of two query heads that share a KV head (so both tiles see the same
// keys), or, where the heads do not pair, two consecutive query blocks of one
// query head group.  One persistent block per SM claims units from a counter;
// eleven warps:
//   warp 0     TMA producer: each unit's Q tiles, then K and V tiles (128
//              keys) into a 2-stage ring, with the column masks of the tiles
//              the mask cuts;
//   warp 1     tcgen05 issuer: S_t = Q_t K^T into TMEM (fp32, 128 lanes x 128
//              columns per tile), and O_t += P_t V with P read from TMEM, one
//              elected thread issuing every MMA;
//   warps 2-9  softmax, one warpgroup per query tile: thread r owns query row
//              r (TMEM lane r).  It reads its S row with tcgen05.ld, applies
//              the mask per element only on tiles the mask cuts, runs the
//              online softmax in base 2, rescales its O row in TMEM when the
//              running maximum has risen by more than 2^8, and writes P (bf16
//              pairs) back over its S columns;
//   warp 10    scheduler: ahead of the others, claims the next unit and lists
//              the key tiles each of its query tiles must visit, classified
//              from precomputed per-tile summaries (which roles, segment
//              numbers and positions occur in a key tile) as hidden (skipped
//              entirely), fully visible (no mask work) or cut by the mask.
// The two query tiles' softmax and MMAs interleave, and consecutive units of
// a block overlap: the next unit's first S products run while the softmax
// warps finish the previous one.
#include <algorithm>
#include <cstddef>
#include <type_traits>

#include "sonic_dev.cuh"
#include "sonic_host.h"

namespace sonic {
namespace {

constexpr int kBM = 128;
constexpr int kBN = 128;
constexpr int kPfThreads = 352;
constexpr int kSchedWarp = 10;
// warps done with a unit slot before the scheduler refills it: the producer
// warp, the issuing thread and the eight softmax warps
constexpr int kUnitConsumers = 10;
constexpr int kMaxKTiles = 2048;
constexpr float kLn2f = 0.6931471805599453f;
constexpr float kLog2ef = 1.4426950408889634f;

// Summary of one 128-row key tile of one sequence.
struct TileSum {
    int32_t flags;     // bit0 body rows, bit1 Nexus rows, bit2 other rows
    int32_t bseg_min;  // segment range of the body rows
    int32_t bseg_max;
    int32_t nseg_min;  // segment range of the Nexus rows
    int32_t nseg_max;
    int32_t n_rows;    // valid key rows in the tile (a prefix of its 128 rows)
    int32_t pos_min;   // S_aug position range of the valid rows
    int32_t pos_max;
};

// Key rows with role 255 are padding (no key): they count as invalid.
// `pos` gives each key row's S_aug position (NULL: the row index itself).
// A k_len outside [0, max_k_len] is refused: the sequence gets no keys.
__device__ __forceinline__ int checked_len(int len, int max_len) {
    return (len < 0 || len > max_len) ? 0 : len;
}

// Rows of sequence (start, len), or 0 when they fall outside [0, total) or
// past max_len: such a sequence is refused, never read.
__device__ __forceinline__ int seq_rows(int start, int len, int max_len, int64_t total) {
    return (start < 0 || (int64_t)start + checked_len(len, max_len) > total) ? 0
                                                                            : checked_len(len, max_len);
}

struct TileMasks;

struct PfParams {
    // query side: the sequences as given (S_aug order)
    const int32_t *k_start, *k_len, *q_start, *q_len;
    const uint8_t *role;
    const int32_t *seg;
    // key side: the same arrays, or their retained-first permutation
    const int32_t *key_start, *key_len;
    const uint8_t *key_role;
    const int32_t *key_seg;
    const int32_t *key_pos;  // S_aug position of each key row; NULL: the row index
    // per key tile of the retained-first order: the first of the 128 consecutive
    // rows of K and V the tile is made of (loaded from them directly), or -1 (the
    // tile is loaded from the permuted copy); NULL in the given order
    const int32_t *key_direct;
    // query chunks of the retained-first query order (query_order_kernel): per
    // sequence qchunks_per_seq words, four per 128-row query tile; NULL: the
    // query rows in the given order
    const int32_t *qchunks;
    int qchunks_per_seq;
    uint16_t *O;
    float *lse;
    float *nexus_mass;
    int32_t *status;
    const TileSum *sums;
    const TileMasks *masks;  // per key tile, from the summary kernel
    int32_t *counter;        // next work unit to claim (zeroed by the summary kernel)
    int n_units, qtiles, HG; // units = qtiles x HG x B x n_layers; HG = Hq >> pack_log2
    int max_k_tiles, max_k_len;
    int B, Hq, G;
    int64_t total_k_rows;  // rows of role, seg_id (and K, V) per layer
    int pack_log2;  // query heads per tile row group: a tile is 128 >> pack_log2 rows x (1 << pack_log2) heads
    int pair;       // 1: a unit's two query tiles are one 128-row block of two query heads
                    // sharing a KV head (else two consecutive 128-row blocks of one)
    int64_t o_ls;
    int o_v8;  // O and its layer stride 32-byte aligned: the epilogue writes whole 32-byte sectors
    int total_q_rows;
    float scale_log2;
    int nexus_mode;
};

// One work unit as the scheduler publishes it.
struct UnitInfo {
    int32_t flags;  // bit 0: no unit is left; bit 1: every query tile visits every listed key tile
    int32_t layer, b, h0, qt;
    int32_t nq;      // query tiles with rows: 1 or 2
    int32_t n_list;  // key tiles listed
    int32_t kstart, klen, kkstart, kklen, qstart, qlen;
    int32_t pbase;    // S_aug position of query row 0 of tile 0
    int32_t last[2];  // list index of the last key tile each query tile visits (-1: none)
    int32_t qc[2][4];  // chunk words of the query tiles (query chunk table)
    int32_t pairu;     // the two query tiles are one block of heads h0 and h0 + 1
    int32_t qstepu;    // query rows between tile 0 and tile 1 (0 when paired)
    int32_t pad[6];
};
static_assert(sizeof(UnitInfo) == 128, "unit record: 128 bytes");

template <int D>
struct PfCfg {
    static constexpr int kHalves = D / 64;
    static constexpr int kQBytes = kBM * D * 2;  // one 128-row Q tile
    static constexpr int kKVBytes = kBN * D * 2;
    static constexpr int kOffQ = 0;                           // [2] Q tiles
    static constexpr int kOffK = kOffQ + 2 * kQBytes;         // [2] stages
    static constexpr int kOffV = kOffK + 2 * kKVBytes;        // [2] stages
    static constexpr int kOffMask = kOffV + 2 * kKVBytes;     // [2] TileMasks
    static constexpr int kOffRole = kOffMask + 2 * 256;       // [2][128] uint8
    static constexpr int kOffSeg = kOffRole + 2 * kBN;        // [2][128] int32
    static constexpr int kOffPos = kOffSeg + 2 * kBN * 4;     // [2][128] int32
    static constexpr int kOffList = kOffPos + 2 * kBN * 4;    // [2 units][kMaxKTiles] int32
    static constexpr int kOffUnit = kOffList + 2 * kMaxKTiles * 4;  // [2] UnitInfo
    static constexpr int kOffBar = kOffUnit + 2 * (int)sizeof(UnitInfo);
    static constexpr int kNumBars = 30;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;   // 16 ints
    static constexpr int kBytes = kOffMisc + 16 * 4;
    static constexpr size_t kSmem = 1024 + kBytes;
};

// Column masks of one 128-key tile (bit c of word w = key 32 w + c of the
// tile): keys that are not body rows (nb), Nexus keys (nx), and the keys of
// each distinct segment among the body keys (bm) and among the Nexus keys
// (nm, used by the causal-segments reading); and the valid keys as runs of
// consecutive S_aug positions (a tile's valid keys are a prefix of its rows
// with increasing positions, so the keys at or before a position form a
// prefix too, whose length the runs give).  With them a row's visibility
// mask costs a few word operations.  More than four distinct segments or
// position runs in one tile set `fallback`: the rule is then evaluated per
// key instead.
struct TileMasks {
    uint32_t nb[4], nx[4];
    int32_t nbody, nnex, fallback, nrun;
    int32_t bseg[4], nseg[4];
    uint32_t bm[4][4], nm[4][4];
    // the valid keys as runs of consecutive S_aug positions, in column order
    int32_t rpos[4], rlen[4];
    int32_t pad[4];
};
static_assert(sizeof(TileMasks) == 256, "tile masks: one 256-byte record per key tile");
static_assert(offsetof(TileMasks, fallback) == 40, "the producer reads fallback as word 10");

// Column of the n-th (from 0) set bit of a 128-bit mask, or -1.
__device__ __forceinline__ int nth_set_bit(const uint32_t m[4], int n) {
    int col = -1;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        const int c = __popc(m[w]);
        if (col < 0 && n < c) {
            uint32_t x = m[w];
            for (int i = 0; i < n; ++i) x &= x - 1;
            col = w * 32 + __ffs(x) - 1;
        }
        if (col < 0) n -= c;
    }
    return col;
}

// The column masks of one key tile, built by one warp: lane l holds key
// 32 w + l of the tile in ro[w], sg[w], ps[w] (role 255, segment 0 and
// position INT_MAX for padding and rows past the sequence).
__device__ __forceinline__ void build_tile_masks(const int (&ro)[4], const int (&sg)[4],
                                                 const int (&ps)[4], int lane, TileMasks *tm) {
    uint32_t bst[4], nst[4], rst[4];
    int pro = 255, psg = 0, pps = INT_MIN, n_valid = 0;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        const bool valid = ro[w] != 255;
        const bool isb = ro[w] == SONIC_ROLE_BODY, isn = ro[w] == SONIC_ROLE_NEXUS;
        const uint32_t nbw = __ballot_sync(0xffffffffu, valid && !isb);
        const uint32_t nxw = __ballot_sync(0xffffffffu, isn);
        n_valid += __popc(__ballot_sync(0xffffffffu, valid));
        // previous key's role/segment/position (lane 0: last key of the
        // previous word)
        int r_up = __shfl_up_sync(0xffffffffu, ro[w], 1);
        int s_up = __shfl_up_sync(0xffffffffu, sg[w], 1);
        int p_up = __shfl_up_sync(0xffffffffu, ps[w], 1);
        if (lane == 0) {
            r_up = pro;
            s_up = psg;
            p_up = pps;
        }
        bst[w] = __ballot_sync(0xffffffffu, isb && !(r_up == SONIC_ROLE_BODY && s_up == sg[w]));
        nst[w] = __ballot_sync(0xffffffffu, isn && !(r_up == SONIC_ROLE_NEXUS && s_up == sg[w]));
        rst[w] = __ballot_sync(0xffffffffu, valid && p_up != ps[w] - 1);
        pro = __shfl_sync(0xffffffffu, ro[w], 31);
        psg = __shfl_sync(0xffffffffu, sg[w], 31);
        pps = __shfl_sync(0xffffffffu, ps[w], 31);
        if (lane == 0) {
            tm->nb[w] = nbw;
            tm->nx[w] = nxw;
        }
    }
    // distinct segments of body runs and Nexus runs (in key order)
    int nb_n = 0, nn_n = 0, fb = 0;
    int bsv[4] = {0, 0, 0, 0}, nsv[4] = {0, 0, 0, 0};
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        uint32_t m = bst[w];
        while (m) {
            const int bl = __ffs(m) - 1;
            m &= m - 1;
            const int v = __shfl_sync(0xffffffffu, sg[w], bl);
            bool seen = false;
#pragma unroll
            for (int k = 0; k < 4; ++k) seen |= (k < nb_n && bsv[k] == v);
            if (!seen) {
                if (nb_n < 4) bsv[nb_n++] = v; else fb = 1;
            }
        }
        m = nst[w];
        while (m) {
            const int bl = __ffs(m) - 1;
            m &= m - 1;
            const int v = __shfl_sync(0xffffffffu, sg[w], bl);
            bool seen = false;
#pragma unroll
            for (int k = 0; k < 4; ++k) seen |= (k < nn_n && nsv[k] == v);
            if (!seen) {
                if (nn_n < 4) nsv[nn_n++] = v; else fb = 1;
            }
        }
    }
#pragma unroll
    for (int k = 0; k < 4; ++k)
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            const uint32_t bmw = __ballot_sync(
                0xffffffffu, k < nb_n && ro[w] == SONIC_ROLE_BODY && sg[w] == bsv[k]);
            const uint32_t nmw = __ballot_sync(
                0xffffffffu, k < nn_n && ro[w] == SONIC_ROLE_NEXUS && sg[w] == nsv[k]);
            if (lane == 0) {
                tm->bm[k][w] = bmw;
                tm->nm[k][w] = nmw;
            }
        }
    const int nrun = __popc(rst[0]) + __popc(rst[1]) + __popc(rst[2]) + __popc(rst[3]);
    if (lane == 0) {
        tm->nbody = nb_n;
        tm->nnex = nn_n;
        tm->nrun = nrun;
        tm->fallback = fb | (nrun > 4);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            tm->bseg[k] = bsv[k];
            tm->nseg[k] = nsv[k];
            tm->pad[k] = 0;
        }
    }
    // position run k (lane k < 4): from the k-th run start to the next one
    // (or to the last valid key); the start's position from the lane holding it
    const int c0 = nth_set_bit(rst, lane & 3), c1 = nth_set_bit(rst, (lane & 3) + 1);
    int start_pos = 0;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        const int v = __shfl_sync(0xffffffffu, ps[w], c0 & 31);
        if (c0 >= 0 && (c0 >> 5) == w) start_pos = v;
    }
    if (lane < 4) {
        tm->rpos[lane] = c0 < 0 ? 0 : start_pos;
        tm->rlen[lane] = c0 < 0 ? 0 : (c1 < 0 ? n_valid : c1) - c0;
    }
}

__global__ void __launch_bounds__(128)
tile_summary_kernel(const uint8_t *__restrict__ role, const int32_t *__restrict__ seg,
                    const int32_t *__restrict__ pos, const int32_t *__restrict__ k_start,
                    const int32_t *__restrict__ k_len, TileSum *__restrict__ out,
                    TileMasks *__restrict__ masks_out, int max_k_tiles, int64_t total_rows,
                    int32_t *status, int32_t *unit_counter) {
    const int t = blockIdx.x, b = blockIdx.y;
    // the attention kernel that follows claims its work units from 0
    if (t == 0 && b == 0 && threadIdx.x == 0) *unit_counter = 0;
    const int len_in = k_len[b];
    // a sequence outside the arrays (or longer than the tiles) gets empty summaries
    const int len = seq_rows(k_start[b], len_in, max_k_tiles * kBN, total_rows);
    if (t == 0 && threadIdx.x == 0 && len != len_in) set_status(status, SONIC_ERR_INVALID_ARGUMENT);
    if (t * kBN >= len && t > 0) return;
    const int r = t * kBN + threadIdx.x;
    int flags = 0, bmin = INT_MAX, bmax = INT_MIN, nmin = INT_MAX, nmax = INT_MIN, n = 0;
    int pmin = INT_MAX, pmax = INT_MIN;
    const int ro = r < len ? role[k_start[b] + r] : 255;
    int sv = 0, pv = INT_MAX;  // padding: no segment, no position
    if (ro != 255) {
        const int s = seg[k_start[b] + r];
        sv = s;
        pv = pos ? pos[k_start[b] + r] : r;
        pmin = pmax = pv;
        n = 1;
        if (ro == SONIC_ROLE_BODY) {
            flags = 1;
            bmin = bmax = s;
        } else if (ro == SONIC_ROLE_NEXUS) {
            flags = 2;
            nmin = nmax = s;
        } else {
            flags = 4;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        flags |= __shfl_xor_sync(0xffffffffu, flags, o);
        bmin = min(bmin, __shfl_xor_sync(0xffffffffu, bmin, o));
        bmax = max(bmax, __shfl_xor_sync(0xffffffffu, bmax, o));
        nmin = min(nmin, __shfl_xor_sync(0xffffffffu, nmin, o));
        nmax = max(nmax, __shfl_xor_sync(0xffffffffu, nmax, o));
        n += __shfl_xor_sync(0xffffffffu, n, o);
        pmin = min(pmin, __shfl_xor_sync(0xffffffffu, pmin, o));
        pmax = max(pmax, __shfl_xor_sync(0xffffffffu, pmax, o));
    }
    __shared__ int sh[4][8];
    const int w = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) {
        sh[w][0] = flags;
        sh[w][1] = bmin;
        sh[w][2] = bmax;
        sh[w][3] = nmin;
        sh[w][4] = nmax;
        sh[w][5] = n;
        sh[w][6] = pmin;
        sh[w][7] = pmax;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        TileSum ts{};
        ts.flags = 0;
        ts.bseg_min = INT_MAX;
        ts.bseg_max = INT_MIN;
        ts.nseg_min = INT_MAX;
        ts.nseg_max = INT_MIN;
        ts.n_rows = 0;
        ts.pos_min = INT_MAX;
        ts.pos_max = INT_MIN;
        for (int i = 0; i < 4; ++i) {
            ts.flags |= sh[i][0];
            ts.bseg_min = min(ts.bseg_min, sh[i][1]);
            ts.bseg_max = max(ts.bseg_max, sh[i][2]);
            ts.nseg_min = min(ts.nseg_min, sh[i][3]);
            ts.nseg_max = max(ts.nseg_max, sh[i][4]);
            ts.n_rows += sh[i][5];
            ts.pos_min = min(ts.pos_min, sh[i][6]);
            ts.pos_max = max(ts.pos_max, sh[i][7]);
        }
        out[(int64_t)b * max_k_tiles + t] = ts;
    }
    // The tile's column masks, built here once per key tile rather than by
    // every block whose query tile the key tile cuts.
    __shared__ int s_ro[kBN], s_sg[kBN], s_ps[kBN];
    s_ro[threadIdx.x] = ro;
    s_sg[threadIdx.x] = sv;
    s_ps[threadIdx.x] = pv;
    __syncthreads();
    if (threadIdx.x < 32) {
        int r4[4], s4[4], p4[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            r4[k] = s_ro[k * 32 + threadIdx.x];
            s4[k] = s_sg[k * 32 + threadIdx.x];
            p4[k] = s_ps[k * 32 + threadIdx.x];
        }
        build_tile_masks(r4, s4, p4, threadIdx.x, masks_out + (int64_t)b * max_k_tiles + t);
    }
}


__device__ __forceinline__ bool visible(int p, int q, int rp, int sp, int rq, int sq,
                                        int mode) {
    if (rq == SONIC_ROLE_BODY) return sq == sp && q <= p;                  // Eqs. 3, 4
    if (rp == SONIC_ROLE_NEXUS && rq == SONIC_ROLE_NEXUS)                  // Eq. 5
        return mode == SONIC_NEXUS_FULL ? true : sq <= sp;
    return q <= p;                                                          // Eq. 3
}

// Largest rise of the running row maximum (base 2) absorbed without
// rescaling O: probabilities stay below 2^8 until the next rescale.
constexpr float kRescaleThreshold = 8.0f;

// The 128-bit visibility mask of query row `pos` (role rp, segment sp) over a
// cut key tile: from the tile's column masks, or per key from its staged
// roles / segments / positions where the masks fall back to the per-key rule.
__device__ __forceinline__ void tile_mask_bits(const TileMasks *tmk, const uint8_t *mrole,
                                               const int32_t *mseg, const int32_t *mpos, int pos,
                                               int rp, int sp, int nexus_mode,
                                               uint32_t (&mbits)[4]) {
    // the whole mask record in independent 16-byte loads
    const uint4 *tv = reinterpret_cast<const uint4 *>(tmk);
    const uint4 nb = tv[0], nx = tv[1], hd = tv[2], bsg = tv[3], nsg = tv[4];
    uint4 bm[4], nm[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        bm[k] = tv[5 + k];
        nm[k] = tv[9 + k];
    }
    if (!hd.z) {
        // causal prefix (keys at or before this row: a prefix of the tile's
        // columns, counted over the position runs), body keys of this row's
        // segment, and the Nexus keys a Nexus row sees
        const uint4 rp4 = tv[13], rl4 = tv[14];
        const int nvis = min(max(pos - (int)rp4.x + 1, 0), (int)rl4.x) +
                         min(max(pos - (int)rp4.y + 1, 0), (int)rl4.y) +
                         min(max(pos - (int)rp4.z + 1, 0), (int)rl4.z) +
                         min(max(pos - (int)rp4.w + 1, 0), (int)rl4.w);
        const int nbody = (int)hd.x, nnex = (int)hd.y;
        const int bs4[4] = {(int)bsg.x, (int)bsg.y, (int)bsg.z, (int)bsg.w};
        const int ns4[4] = {(int)nsg.x, (int)nsg.y, (int)nsg.z, (int)nsg.w};
        uint4 bw = make_uint4(0u, 0u, 0u, 0u), xw = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if (k < nbody && bs4[k] == sp) {
                bw.x |= bm[k].x; bw.y |= bm[k].y; bw.z |= bm[k].z; bw.w |= bm[k].w;
            }
            if (rp == SONIC_ROLE_NEXUS && nexus_mode != SONIC_NEXUS_FULL && k < nnex &&
                ns4[k] <= sp) {
                xw.x |= nm[k].x; xw.y |= nm[k].y; xw.z |= nm[k].z; xw.w |= nm[k].w;
            }
        }
        if (rp == SONIC_ROLE_NEXUS && nexus_mode == SONIC_NEXUS_FULL) xw = nx;
        const uint32_t nbw[4] = {nb.x, nb.y, nb.z, nb.w};
        const uint32_t bww[4] = {bw.x, bw.y, bw.z, bw.w};
        const uint32_t xww[4] = {xw.x, xw.y, xw.z, xw.w};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            const int nw = min(max(nvis - 32 * w, 0), 32);
            const uint32_t cw = nw >= 32 ? 0xffffffffu : ((1u << nw) - 1u);
            mbits[w] = (cw & (nbw[w] | bww[w])) | xww[w];
        }
    } else {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const uint8_t *mr = mrole + c * 32;
            const int32_t *ms = mseg + c * 32;
            const int32_t *mp = mpos + c * 32;
            uint32_t bits = 0;
#pragma unroll 4
            for (int e = 0; e < 32; ++e) {
                const int rq = mr[e];
                const bool v = rq != 255 && visible(pos, mp[e], rp, sp, rq, ms[e], nexus_mode);
                bits |= (v ? 1u : 0u) << e;
            }
            mbits[c] = bits;
        }
    }
}

// One persistent block per SM walks work units: a unit is two 128-row query
// tiles of one (layer, sequence).  Paired (pair = 1: unpacked heads, an even
// number per KV head): one query block of heads h0 (tile 0) and h0 + 1
// (tile 1), whose key-tile lists are then the same.  Otherwise: rows 0..127
// (tile 0) and 128..255 (tile 1) of a 256-row block of one query-head group.
// Eleven warps (352 threads):
//   warp 0       TMA producer: the unit's Q tiles, then K, V (and the key
//                metadata of cut tiles) into a 2-stage ring that runs on
//                across units;
//   warp 1       tcgen05 issuer and TMEM owner;
//   warps 2-5    softmax of query tile 0, warps 6-9 of query tile 1 (warp w
//                reaches TMEM lanes 32 * (w % 4) .. + 31);
//   warp 10      scheduler: claims the next unit from a counter, summarises
//                its query tiles and lists the key tiles each of them must
//                visit, up to two units ahead of the others.
// TMEM (512 columns): S/P of tile 0 at 0, of tile 1 at 128, O of tile 0 at
// 256, O of tile 1 at 384.  P (bf16 pairs) overwrites the first 64 columns of
// its S block and feeds O += P V straight from tensor memory.  While the
// softmax warps finish one unit (normalise O, write it out), the issuer
// already runs the next unit's first S products: O is overwritten only after
// the epilogue has read it (o_free), S/P only after the last P.V read it (the
// tensor pipe runs in order).
// kOut: bit 0 writes the log-sum-exp, bit 1 the attention mass on Nexus keys.
// kQC: the query tiles come from the chunk table of the retained-first query
// order (query_order_kernel) instead of consecutive query rows.
// kSolo: every unit has one query tile (packed heads, short query blocks).  Its
// S/P then alternates between the two tiles' TMEM blocks, so the S product of
// key tile j + 1 runs while the softmax works on tile j, and K takes a ring of
// three stages (the unused second Q tile's buffer is the third), V of two.
// kPair: paired units (an even number of query heads per KV head, heads not
// packed): a unit is one 128-row query block of heads h0 and h0 + 1.
template <int D, int kOut, bool kQC, bool kSolo, bool kPair>
__global__ void __maxnreg__(168)
prefill_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
               const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmK0,
               const __grid_constant__ CUtensorMap tmV0, const __grid_constant__ CUtensorMap tmQ32,
               const PfParams p) {
    using C = PfCfg<D>;
    constexpr bool kLse = kOut & 1, kMass = kOut & 2;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t *Qs = smem + C::kOffQ;
    uint8_t *Ks = smem + C::kOffK;
    uint8_t *Vs = smem + C::kOffV;
    TileMasks *tmasks = reinterpret_cast<TileMasks *>(smem + C::kOffMask);
    uint8_t *meta_role = smem + C::kOffRole;
    int32_t *meta_seg = reinterpret_cast<int32_t *>(smem + C::kOffSeg);
    int32_t *meta_pos = reinterpret_cast<int32_t *>(smem + C::kOffPos);
    int32_t *lists = reinterpret_cast<int32_t *>(smem + C::kOffList);  // [2][kMaxKTiles]
    UnitInfo *units = reinterpret_cast<UnitInfo *>(smem + C::kOffUnit);  // [2]
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + C::kOffBar);
    uint64_t *q_full = bars + 0;
    uint64_t *q_empty = bars + 1;
    uint64_t *kv_full = bars + 2;     // [2] per ring stage
    uint64_t *kv_empty = bars + 4;    // [2]
    // [stage][query tile]: key metadata of a stage written, for a query tile
    // that reads it (the key tile cuts the query tile, or has some Nexus keys
    // and the Nexus mass is asked for).  A phase completes only for such
    // tiles, so each softmax warpgroup waits every phase of its own barrier
    // in turn, whatever key tiles it skips.
    uint64_t *meta_full = bars + 6;   // [2][2]
    uint64_t *s_full = bars + 10;     // [2] per query tile
    uint64_t *p_full = bars + 12;     // [2]
    uint64_t *o_done = bars + 14;     // [2]
    uint64_t *o_free = bars + 16;     // [2]
    uint64_t *unit_full = bars + 18;  // [2] per unit slot
    uint64_t *unit_empty = bars + 20; // [2]
    uint64_t *mma_idle = bars + 22;
    // kSolo only: K ring stages (written / free again), and one P.V product done
    uint64_t *k_full = bars + 23;   // [3]
    uint64_t *k_empty = bars + 26;  // [3]
    uint64_t *pv_done = bars + 29;
    int32_t *misc = reinterpret_cast<int32_t *>(smem + C::kOffMisc);
    // misc: 0 tmem base, 2 abort
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + 2);

    // A query tile is R query rows x P heads of one KV group (P = 1 << pack_log2,
    // R = 128 / P): tile row r is query row r / P, head h0 + r % P.  P > 1 packs
    // the heads of short query blocks so the tile rows are not left empty.
    const int pl2 = p.pack_log2, R = kBM >> pl2;
    // query rows of a unit, and the row offset of its second query tile
    const int urows = kPair ? R : 2 * R, qstep = kPair ? 0 : R;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        mbar_init(q_full, 1);
        mbar_init(q_empty, 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(&kv_full[s], 1);
            mbar_init(&kv_empty[s], 1);
            mbar_init(&meta_full[2 * s], 1);
            mbar_init(&meta_full[2 * s + 1], 1);
            mbar_init(&s_full[s], 1);
            mbar_init(&p_full[s], kBM);
            mbar_init(&o_done[s], 1);
            mbar_init(&o_free[s], kBM);
            mbar_init(&unit_full[s], 1);
            mbar_init(&unit_empty[s], kUnitConsumers);
        }
        mbar_init(mma_idle, 1);
        if (kSolo) {
            for (int s = 0; s < 3; ++s) {
                mbar_init(&k_full[s], 1);
                mbar_init(&k_empty[s], 1);
            }
            mbar_init(pv_done, 1);
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(reinterpret_cast<uint32_t *>(&misc[0]), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = static_cast<uint32_t>(misc[0]);
    // what the producer issued, for the drain after an abort
    int issued_q = 0, issued_kv = 0, issued_k = 0;

    if (warp == kSchedWarp) {
        // ------------------------------------------------------------ scheduler
        for (int k = 0;; ++k) {
            const int slot = k & 1;
            int end = 0, layer = 0, b = 0, hg = 0, qt = 0, cw = 0;
            bool lpair = false;  // a last query block shared by two heads (below)
            int kstart = 0, klen = 0, qstart = 0, qlen = 0, kkstart = 0, kklen = 0;
            for (;;) {
                int u = p.n_units;
                if (lane == 0 && !*abort_flag && !timed_out(p.status)) u = atomicAdd(p.counter, 1);
                u = __shfl_sync(0xffffffffu, u, 0);
                if (u >= p.n_units) {
                    end = 1;
                    break;
                }
                // units: query-head group fastest, then query block (the last
                // first: the longest lists go first), then sequence, then layer;
                // the blocks running together read one sequence's K/V, which
                // stays in L2
                hg = u % p.HG;
                int rest = u / p.HG;
                qt = p.qtiles - 1 - rest % p.qtiles;
                rest /= p.qtiles;
                b = rest % p.B;
                layer = rest / p.B;
                klen = p.k_len[b];
                qlen = p.q_len[b];
                kstart = p.k_start[b];
                qstart = p.q_start[b];
                if (kstart < 0 || (int64_t)kstart + klen > p.total_k_rows || qstart < 0 ||
                    qlen < 0 || (int64_t)qstart + qlen > p.total_q_rows) {
                    // rows outside the arrays: the sequence is refused, nothing is read
                    if (lane == 0 && hg == 0 && qt == 0) set_status(p.status, SONIC_ERR_INVALID_ARGUMENT);
                    continue;
                }
                if constexpr (kQC) {
                    // lane l < 8: chunk l & 3 of query tile l >> 2 (paired: both
                    // tiles are the same rows)
                    cw = 0;
                    if (lane < 8) {
                        const int vt = kPair ? qt : 2 * qt + (lane >> 2);
                        if ((vt + 1) * 4 <= p.qchunks_per_seq)
                            cw = p.qchunks[(int64_t)b * p.qchunks_per_seq + vt * 4 + (lane & 3)];
                    }
                    if (!__any_sync(0xffffffffu, (cw >> 24) != 0)) continue;  // no query rows
                } else {
                    if (qt * urows >= qlen) continue;  // no query rows in this block
                    // Unpaired units (an odd head ratio) are 256-row blocks of one head;
                    // the last block of a sequence with an odd number of 128-row blocks
                    // has one tile, and one tile alone leaves the tensor pipe idle
                    // during its softmax.  Heads 2i and 2i + 1 of a KV group share that
                    // block instead (same rows, same keys: the paired form); the last
                    // head of an odd group keeps a unit of its own.
                    lpair = false;
                    if (!kSolo && !kPair && pl2 == 0 && p.G > 1 && qt * urows + R >= qlen) {
                        const int i = hg % p.G;
                        if (i & 1) continue;  // in the unit of head hg - 1
                        lpair = i + 1 < p.G;
                    }
                }
                kklen = p.key_len[b];
                if (qlen > klen || klen > p.max_k_len || kklen > p.max_k_tiles * kBN) {
                    // the host-side bounds were wrong for this sequence: refuse it
                    if (lane == 0) set_status(p.status, SONIC_ERR_INVALID_ARGUMENT);
                    continue;
                }
                kkstart = p.key_start[b];
                break;
            }
            // The slot is free once every consumer is done with unit k - 2.  A
            // unit takes microseconds: poll sparingly (a sleeping warp leaves
            // its scheduler's issue slots to the softmax warps), then wait.
            if (k >= 2) {
                const uint32_t par = ((k >> 1) - 1) & 1;
                const uint64_t t0 = global_ns();
                while (!mbar_test(&unit_empty[slot], par) && !*abort_flag &&
                       global_ns() - t0 < SONIC_WAIT_LIMIT_NS)
                    __nanosleep(500);
                if (!mbar_wait(&unit_empty[slot], par, p.status, abort_flag)) break;
            }
            UnitInfo *ui = units + slot;
            if (end) {
                if (lane == 0) {
                    ui->flags = 1;
                    mbar_arrive(&unit_full[slot]);
                }
                break;
            }
            const int pbase = klen - qlen + qt * urows;  // position of query row 0 of tile 0
            // summaries of the query tiles: S_aug position range (smallest and
            // largest), segment range, Nexus rows and their segment range
            int qf[2], qs0[2], qs1[2], qn0[2], qn1[2], qp0[2], qp1[2];
            bool tile1;
            if constexpr (kQC) {
                // Chunk words (lane l < 8: chunk l & 3 of tile l >> 2) turned into
                // (query rows << 24) | S_aug position of the chunk's first row;
                // tile row r is row r & 31 of chunk r >> 5.
                cw = (cw & ~0xffffff) | (klen - qlen + (cw & 0xffffff));
#pragma unroll
                for (int qi = 0; qi < 2; ++qi) {
                    int f = 0, s0 = INT_MAX, s1 = INT_MIN, n0 = INT_MAX, n1 = INT_MIN;
                    int pmin = INT_MAX, pmax = INT_MIN;
#pragma unroll
                    for (int c = 0; c < kBM / 32; ++c) {
                        const int w = __shfl_sync(0xffffffffu, cw, qi * 4 + c);
                        const int pos = (w & 0xffffff) + lane;
                        if (lane < (w >> 24)) {
                            const int ro = p.role[kstart + pos];
                            const int s = p.seg[kstart + pos];
                            pmin = min(pmin, pos);
                            pmax = max(pmax, pos);
                            s0 = min(s0, s);
                            s1 = max(s1, s);
                            if (ro == SONIC_ROLE_NEXUS) {
                                f = 2;
                                n0 = min(n0, s);
                                n1 = max(n1, s);
                            }
                        }
                    }
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) {
                        f |= __shfl_xor_sync(0xffffffffu, f, o);
                        s0 = min(s0, __shfl_xor_sync(0xffffffffu, s0, o));
                        s1 = max(s1, __shfl_xor_sync(0xffffffffu, s1, o));
                        n0 = min(n0, __shfl_xor_sync(0xffffffffu, n0, o));
                        n1 = max(n1, __shfl_xor_sync(0xffffffffu, n1, o));
                        pmin = min(pmin, __shfl_xor_sync(0xffffffffu, pmin, o));
                        pmax = max(pmax, __shfl_xor_sync(0xffffffffu, pmax, o));
                    }
                    qf[qi] = f;
                    qs0[qi] = s0;
                    qs1[qi] = s1;
                    qn0[qi] = n0;
                    qn1[qi] = n1;
                    qp0[qi] = pmin;
                    qp1[qi] = pmax;
                }
                tile1 = kPair || qp0[1] <= qp1[1];
            } else {
                tile1 = kPair || (!kPair && lpair) || qt * 2 * R + R < qlen;
#pragma unroll
                for (int qi = 0; qi < 2; ++qi) {
                    int f = 0, s0 = INT_MAX, s1 = INT_MIN, n0 = INT_MAX, n1 = INT_MIN;
                    for (int r = lane; r < R; r += 32) {
                        const int pos = pbase + qi * (lpair ? 0 : qstep) + r;
                        if (pos <= klen - 1) {
                            const int ro = p.role[kstart + pos];
                            const int s = p.seg[kstart + pos];
                            s0 = min(s0, s);
                            s1 = max(s1, s);
                            if (ro == SONIC_ROLE_NEXUS) {
                                f = 2;
                                n0 = min(n0, s);
                                n1 = max(n1, s);
                            }
                        }
                    }
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) {
                        f |= __shfl_xor_sync(0xffffffffu, f, o);
                        s0 = min(s0, __shfl_xor_sync(0xffffffffu, s0, o));
                        s1 = max(s1, __shfl_xor_sync(0xffffffffu, s1, o));
                        n0 = min(n0, __shfl_xor_sync(0xffffffffu, n0, o));
                        n1 = max(n1, __shfl_xor_sync(0xffffffffu, n1, o));
                    }
                    qf[qi] = f;
                    qs0[qi] = s0;
                    qs1[qi] = s1;
                    qn0[qi] = n0;
                    qn1[qi] = n1;
                    qp0[qi] = pbase + qi * (lpair ? 0 : qstep);
                    qp1[qi] = min(qp0[qi] + R - 1, klen - 1);
                }
            }
            // Key tiles to visit: a key tile is listed when either query tile
            // sees some of it.  entry: (tile << 6) | (Nexus keys: 0 none, 1 all,
            // 2 some) << 4 | (tile 1 sees it) << 3 | (tile 0 sees it) << 2
            // | (not all of it visible to tile 1) << 1 | (... to tile 0)
            int32_t *lst = lists + slot * kMaxKTiles;
            const int n_kt = (kklen + kBN - 1) / kBN;
            int n_list = 0, last0 = -1, last1 = -1, skipped = 0;
            for (int c0 = 0; c0 < n_kt; c0 += 32) {
                const int t = c0 + lane;
                int entry = 0;
                bool need[2] = {false, false};
                if (t < n_kt) {
                    const TileSum ts = p.sums[(int64_t)b * p.max_k_tiles + t];
                    const int k0 = ts.pos_min, k1 = ts.pos_max;  // S_aug positions of the keys
                    const bool kb = ts.flags & 1, kn = ts.flags & 2, ko = ts.flags & 4;
                    entry = (t << 6) | ((kn ? ((kb || ko) ? 2 : 1) : 0) << 4);
#pragma unroll
                    for (int qi = 0; qi < 2; ++qi) {
                        // S_aug positions of the query tile's rows: smallest, largest
                        const int p0 = qp0[qi], p1 = qp1[qi];
                        if (p0 > p1) continue;
                        const bool q_has_nexus = qf[qi] & 2;
                        const bool causal_part = (k0 <= p1) && (kn || ko);
                        const bool body_part =
                            kb && (k0 <= p1) && !(ts.bseg_max < qs0[qi] || ts.bseg_min > qs1[qi]);
                        const bool nexus_part =
                            kn && q_has_nexus &&
                            (p.nexus_mode == SONIC_NEXUS_FULL || ts.nseg_min <= qn1[qi]);
                        const bool any = causal_part || body_part || nexus_part;
                        const bool full =
                            any && ts.n_rows == kBN && k1 <= p0 &&
                            (!kb || (ts.bseg_min == ts.bseg_max && qs0[qi] == qs1[qi] &&
                                     ts.bseg_min == qs0[qi])) &&
                            (p.nexus_mode == SONIC_NEXUS_FULL || !(kn && q_has_nexus) ||
                             ts.nseg_max <= qn0[qi]);
                        need[qi] = any;
                        if (any) entry |= 4 << qi;
                        if (!full) entry |= 1 << qi;
                    }
                }
                const bool keep = need[0] || need[1];
                const unsigned bal = __ballot_sync(0xffffffffu, keep);
                skipped += __popc(__ballot_sync(0xffffffffu, keep && !need[0])) +
                           (tile1 ? __popc(__ballot_sync(0xffffffffu, keep && !need[1])) : 0);
                const unsigned b0 = __ballot_sync(0xffffffffu, need[0]);
                const unsigned b1 = __ballot_sync(0xffffffffu, need[1]);
                if (keep) lst[n_list + __popc(bal & ((1u << lane) - 1u))] = entry;
                // list index of the last entry each query tile visits
                if (b0) last0 = n_list + __popc(bal & ((2u << (31 - __clz(b0))) - 1u)) - 1;
                if (b1) last1 = n_list + __popc(bal & ((2u << (31 - __clz(b1))) - 1u)) - 1;
                n_list += __popc(bal);
            }
            // both query tiles visit every listed key tile (masked where they see
            // none of it) unless skipping drops more than a tenth of the products
            const bool dense = skipped * 10 <= (tile1 ? 2 : 1) * n_list;
            if (lane == 0) {
                ui->flags = dense ? 2 : 0;
                ui->layer = layer;
                ui->b = b;
                ui->h0 = kPair ? 2 * hg : hg << pl2;
                if (!kPair) {
                    ui->pairu = lpair;
                    ui->qstepu = lpair ? 0 : qstep;
                }
                ui->qt = qt;
                ui->nq = tile1 ? 2 : 1;
                ui->n_list = n_list;
                ui->kstart = kstart;
                ui->klen = klen;
                ui->kkstart = kkstart;
                ui->kklen = kklen;
                ui->qstart = qstart;
                ui->qlen = qlen;
                ui->pbase = pbase;
                ui->last[0] = last0;
                ui->last[1] = last1;
            }
            if (kQC && lane < 8) ui->qc[lane >> 2][lane & 3] = cw;
            // every lane's list entries are written before lane 0 publishes the slot
            __syncwarp();
            if (lane == 0) mbar_arrive(&unit_full[slot]);
        }
    } else if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&tmQ);
            tma_prefetch_desc(&tmK);
            tma_prefetch_desc(&tmV);
            if (p.key_direct != nullptr) {
                tma_prefetch_desc(&tmK0);
                tma_prefetch_desc(&tmV0);
            }
            if (p.qchunks != nullptr) tma_prefetch_desc(&tmQ32);
        }
        int g = 0;  // K/V tiles issued over all units (ring position)
        bool ok = true;
        for (int k = 0; ok; ++k) {
            const int slot = k & 1;
            if (!mbar_wait(&unit_full[slot], (k >> 1) & 1, p.status, abort_flag)) break;
            const UnitInfo *ui = units + slot;
            if (ui->flags & 1) break;
            const int n_list = ui->n_list, nq = ui->nq, layer = ui->layer, b = ui->b;
            const int kkstart = ui->kkstart, kklen = ui->kklen;
            const bool udense = ui->flags & 2;  // both query tiles visit every listed tile
            const int32_t *lst = lists + slot * kMaxKTiles;
            if (n_list > 0) {
                // Q: its buffer is free once the previous unit's last S products are done
                if (issued_q > 0 &&
                    !mbar_wait(q_empty, (issued_q - 1) & 1, p.status, abort_flag))
                    break;
                if (kQC && lane == 0) {
                    // a query tile of 128 consecutive query rows in one copy, any
                    // other from its 32-row chunks (a chunk without rows is not
                    // loaded: its tile rows are computed and never written)
                    const int q0 = ui->qstart - (ui->klen - ui->qlen);  // Q row of position 0
                    int bytes = 0;
                    bool whole[2] = {false, false};
#pragma unroll
                    for (int qi = 0; qi < 2; ++qi) {
                        if (qi >= nq) break;
                        const int w0 = ui->qc[qi][0];
                        whole[qi] = true;
#pragma unroll
                        for (int c = 0; c < kBM / 32; ++c) {
                            const int w = ui->qc[qi][c];
                            whole[qi] = whole[qi] && w == w0 + c * 32;
                            if ((w >> 24) != 0) bytes += 32 * D * 2;
                        }
                        whole[qi] = whole[qi] && (w0 >> 24) == 32;
                    }
                    mbar_arrive_expect_tx(q_full, bytes);
#pragma unroll
                    for (int qi = 0; qi < 2; ++qi) {
                        if (qi >= nq) break;
                        if (whole[qi]) {
                            // both 64-column halves in one copy (5-D map: the half is a
                            // dimension of its own, outside the rows)
                            tma_load_5d(Qs + qi * C::kQBytes, &tmQ, q_full, 0,
                                        ui->h0 + qi * (kPair ? 1 : 0),
                                        q0 + (ui->qc[qi][0] & 0xffffff), 0, layer);
                            continue;
                        }
#pragma unroll
                        for (int c = 0; c < kBM / 32; ++c) {
                            const int w = ui->qc[qi][c];
                            if ((w >> 24) == 0) continue;
#pragma unroll
                            for (int hh = 0; hh < C::kHalves; ++hh)
                                tma_load_4d(Qs + qi * C::kQBytes + hh * (kBM * 128) + c * (32 * 128),
                                            &tmQ32, q_full, hh * 64, ui->h0 + qi * (kPair ? 1 : 0),
                                            q0 + (w & 0xffffff), layer);
                        }
                    }
                } else if (!kQC && lane == 0) {
                    mbar_arrive_expect_tx(q_full, nq * C::kQBytes);
                    for (int qi = 0; qi < nq; ++qi)
                        tma_load_5d(Qs + qi * C::kQBytes, &tmQ, q_full, 0,
                                    ui->h0 + qi * (kPair ? 1 : ui->pairu),
                                    ui->qstart + ui->qt * urows + qi * (kPair ? 0 : ui->qstepu), 0,
                                    layer);
                }
                ++issued_q;
                const int kvh = ui->h0 / p.G;
                // The key tile's column masks (built once per key tile by the summary
                // kernel; 8 bytes per lane), where a query tile is cut or the Nexus
                // mass needs the Nexus bits, into the metadata of ring stage st; the
                // keys' roles / segments / S_aug positions only where the masks fall
                // back to the per-key rule.
                auto stage_meta = [&](int st, int e, bool need_m0, bool need_m1) {
                    const int kt = e >> 6;
                    const bool cut_any = (e & 3) != 0;
                    if (need_m0 || need_m1) {
                        const uint2 mw = reinterpret_cast<const uint2 *>(
                            p.masks + (int64_t)b * p.max_k_tiles + kt)[lane];
                        reinterpret_cast<uint2 *>(tmasks + st)[lane] = mw;
                        // word 10 of the record (lane 5's first word): fallback
                        const int fallback = __shfl_sync(0xffffffffu, (int)mw.x, 5);
                        if (cut_any && fallback) {
                            int ro[4], sg[4], ps[4];
                            // all twelve loads first, none waiting on another
#pragma unroll
                            for (int w = 0; w < 4; ++w) {
                                const int q = kt * kBN + w * 32 + lane;
                                const bool in = q < kklen;
                                ro[w] = in ? p.key_role[kkstart + q] : 255;
                                sg[w] = in ? p.key_seg[kkstart + q] : 0;
                                ps[w] = in ? (p.key_pos != nullptr ? p.key_pos[kkstart + q] : q)
                                           : INT_MAX;
                            }
#pragma unroll
                            for (int w = 0; w < 4; ++w) {
                                const int c = w * 32 + lane;
                                const bool pad = ro[w] == 255;  // no segment, no position
                                meta_role[st * kBN + c] = (uint8_t)ro[w];
                                meta_seg[st * kBN + c] = pad ? 0 : sg[w];
                                meta_pos[st * kBN + c] = pad ? INT_MAX : ps[w];
                            }
                        }
                        // every lane's metadata is written before lane 0 releases it
                        __syncwarp();
                        if (lane == 0) {
                            if (need_m0) mbar_arrive(&meta_full[2 * st]);
                            if (need_m1) mbar_arrive(&meta_full[2 * st + 1]);
                        }
                    }
                };
                // a retained-first tile made of 128 consecutive input rows is copied
                // from K and V themselves (the load overlaps the wait that follows)
                auto src_of = [&](int kt) {
                    return p.key_direct != nullptr
                               ? p.key_direct[(int64_t)b * p.max_k_tiles + kt]
                               : -1;
                };
                if constexpr (kSolo) {
                    // One query tile: K of key tile i + 1 is copied before V of tile
                    // i, into a ring of three stages (Ks, Ks + one stage, and the
                    // second Q tile's buffer), V into a ring of two; key tile i's
                    // metadata goes with its V stage.
                    int gk = g;
                    auto issue_k = [&](int i) -> bool {
                        const int kt = lst[i] >> 6;
                        const int dsrc = src_of(kt);
                        const int ks = gk % 3;
                        if (gk >= 3 &&
                            !mbar_wait(&k_empty[ks], ((gk / 3) - 1) & 1, p.status, abort_flag))
                            return false;
                        if (lane == 0) {
                            mbar_arrive_expect_tx(&k_full[ks], C::kKVBytes);
                            uint8_t *dst = ks < 2 ? Ks + ks * C::kKVBytes : Qs + C::kQBytes;
                            tma_load_5d(dst, dsrc >= 0 ? &tmK0 : &tmK, &k_full[ks], 0, kvh,
                                        dsrc >= 0 ? dsrc : kkstart + kt * kBN, 0, layer);
                        }
                        issued_k = ++gk;
                        return true;
                    };
                    if (!issue_k(0)) ok = false;
                    for (int i = 0; ok && i < n_list; ++i, ++g) {
                        if (i + 1 < n_list && !issue_k(i + 1)) {
                            ok = false;
                            break;
                        }
                        const int st = g & 1;
                        const int e = lst[i];
                        const int kt = e >> 6;
                        const int dsrc = src_of(kt);
                        if (g >= 2 &&
                            !mbar_wait(&kv_empty[st], ((g >> 1) - 1) & 1, p.status, abort_flag)) {
                            ok = false;
                            break;
                        }
                        if (lane == 0) {
                            mbar_arrive_expect_tx(&kv_full[st], C::kKVBytes);
                            tma_load_5d(Vs + st * C::kKVBytes, dsrc >= 0 ? &tmV0 : &tmV,
                                        &kv_full[st], 0, kvh, dsrc >= 0 ? dsrc : kkstart + kt * kBN,
                                        0, layer);
                        }
                        issued_kv = g + 1;
                        stage_meta(st, e, (e & 1) || (kMass && ((e >> 4) & 3) == 2), false);
                    }
                } else {
                    for (int i = 0; i < n_list; ++i, ++g) {
                        const int st = g & 1;
                        const int e = lst[i];
                        const int kt = e >> 6;
                        const int dsrc = src_of(kt);
                        if (g >= 2 &&
                            !mbar_wait(&kv_empty[st], ((g >> 1) - 1) & 1, p.status, abort_flag)) {
                            ok = false;
                            break;
                        }
                        // query tiles visiting the key tile that read its metadata: cut
                        // by the mask, or (Nexus mass) some of its keys are Nexus keys
                        const bool mass_tile = kMass && ((e >> 4) & 3) == 2;
                        const bool need_m0 = (udense || (e & 4)) && ((e & 1) || mass_tile);
                        const bool need_m1 =
                            nq == 2 && (udense || (e & 8)) && ((e & 2) || mass_tile);
                        // K/V copies first; the key metadata is built while they are in
                        // flight and has a barrier of its own, so the S product of a cut
                        // tile waits for the copy alone
                        if (lane == 0) {
                            mbar_arrive_expect_tx(&kv_full[st], 2 * C::kKVBytes);
                            const bool direct = dsrc >= 0;
                            const int row = direct ? dsrc : kkstart + kt * kBN;
                            const CUtensorMap *mk = direct ? &tmK0 : &tmK;
                            const CUtensorMap *mv = direct ? &tmV0 : &tmV;
                            tma_load_5d(Ks + st * C::kKVBytes, mk, &kv_full[st], 0, kvh, row, 0,
                                        layer);
                            tma_load_5d(Vs + st * C::kKVBytes, mv, &kv_full[st], 0, kvh, row, 0,
                                        layer);
                        }
                        issued_kv = g + 1;
                        stage_meta(st, e, need_m0, need_m1);
                    }
                }
            }
            if (!ok) break;
            __syncwarp();
            if (lane == 0) mbar_arrive(&unit_empty[slot]);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        // This thread is on the path of every key tile, so its loop is
        // specialised on the number of query tiles and on whether both visit
        // every listed key tile (no per-tile checks then), and each descriptor
        // is a per-stage word plus a constant: an MMA then costs about two
        // instructions besides itself.
        if (lane == 0) {
            constexpr uint32_t idS = idesc_bf16_f32(kBM, kBN, 0);
            constexpr uint32_t idPV = idesc_bf16_f32(kBM, D, 1);
            constexpr uint32_t dhi = sw128_desc_hi(1024);
            const uint32_t q_lo = sw128_desc_lo(smem_u32(Qs), 16);
            const uint32_t k_lo = sw128_desc_lo(smem_u32(Ks), 16);
            const uint32_t v_lo = sw128_desc_lo(smem_u32(Vs), kBN * 128);
            // S_qi = Q_qi K^T from the K stage whose descriptor word is kst
            auto issue_s = [&](int qi, uint32_t kst) {
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t off = ((kk >> 2) * (kBM * 128) + (kk & 3) * 32) >> 4;
                    tc_mma_ss(tmem + qi * kBN,
                              desc_join(q_lo + ((qi * C::kQBytes) >> 4) + off, dhi),
                              desc_join(kst + off, dhi), idS, kk > 0 ? 1u : 0u);
                }
                tc_commit(&s_full[qi]);
            };
            // O_qi (+)= P_qi V from the V stage whose descriptor word is vst (P over
            // the first columns of S_qi)
            auto issue_pv = [&](int qi, uint32_t vst, bool acc0) {
#pragma unroll
                for (int kk = 0; kk < kBN / 16; ++kk)
                    tc_mma_ts(tmem + 256 + qi * 128, tmem + qi * kBN + kk * 8,
                              desc_join(vst + ((kk * (16 * 128)) >> 4), dhi), idPV,
                              (acc0 || kk > 0) ? 1u : 0u);
            };
            // descriptor words of K and V in ring stage st
            constexpr uint32_t kStageStep = C::kKVBytes >> 4;
            auto k_of = [&](int st) { return k_lo + (st ? kStageStep : 0u); };
            auto v_of = [&](int st) { return v_lo + (st ? kStageStep : 0u); };
            int g = 0, nqu = 0;          // ring position; units with work so far
            uint32_t pw[2] = {0u, 0u};   // P phases waited per query tile
            int uo[2] = {0, 0};          // units whose O each query tile accumulated
            bool ok = true;
            for (int k = 0; ok; ++k) {
                const int slot = k & 1;
                if (!mbar_wait(&unit_full[slot], (k >> 1) & 1, p.status, abort_flag)) break;
                const UnitInfo *ui = units + slot;
                if (ui->flags & 1) break;
                const int n_list = ui->n_list, nq = ui->nq;
                const int last[2] = {ui->last[0], ui->last[1]};
                const int32_t *lst = lists + slot * kMaxKTiles;
                if (n_list > 0) {
                    ok = mbar_wait(q_full, nqu & 1, p.status, abort_flag);
                    ++nqu;
                    // Key tile j (ring stage (g + j) & 1): P.V of each query tile
                    // visiting it, then that tile's S of the next key tile it
                    // visits.  The tensor pipe runs in order, so the next S never
                    // overwrites a P still being read.
                    // DENSE: every query tile visits every listed key tile (no list
                    // reads or per-tile checks on this thread's path)
                    auto run = [&](auto nq_tag, auto dense_tag) -> bool {
                        constexpr int NQ = decltype(nq_tag)::value;
                        constexpr bool DENSE = decltype(dense_tag)::value;
                        auto visits = [&](int ent, int qi) -> bool {
                            return DENSE || ((ent >> (2 + qi)) & 1);
                        };
                        bool first[2] = {true, true};
                        int e = DENSE ? 0 : lst[0];
                        int en = (DENSE || n_list < 2) ? 0 : lst[1];
                        if (!mbar_wait(&kv_full[g & 1], (g >> 1) & 1, p.status, abort_flag))
                            return false;
                        tc_fence_after();
#pragma unroll
                        for (int qi = 0; qi < NQ; ++qi)
                            if (visits(e, qi)) issue_s(qi, k_of(g & 1));
                        if (n_list == 1) tc_commit(q_empty);
                        // key tile j sits in ring stage (g + j) & 1; one copy of the
                        // body, the stage entering only through descriptor words
                        for (int j = 0; j < n_list; ++j) {
                            const int ST = (g + j) & 1;
                            const uint32_t vst = v_of(ST), kst_next = k_of(ST ^ 1);
                            const bool more = j + 1 < n_list;
                            // the entry after next, loaded a tile ahead of its use
                            const int enn = (DENSE || j + 2 >= n_list) ? 0 : lst[j + 2];
                            const int lastq = DENSE ? NQ - 1 : ((NQ == 2 && ((e >> 3) & 1)) ? 1 : 0);
                            bool kv_ready = false;
#pragma unroll
                            for (int qi = 0; qi < NQ; ++qi) {
                                if (visits(e, qi)) {
                                    if (!mbar_wait(&p_full[qi], pw[qi] & 1, p.status, abort_flag))
                                        return false;
                                    ++pw[qi];
                                    tc_fence_after();
                                    const bool fst = DENSE ? j == 0 : first[qi];
                                    if (fst && uo[qi] > 0) {
                                        // O still holds the previous unit until its
                                        // epilogue has read it
                                        if (!mbar_wait(&o_free[qi], (uo[qi] - 1) & 1, p.status,
                                                       abort_flag))
                                            return false;
                                        tc_fence_after();
                                    }
                                    issue_pv(qi, vst, !fst);
                                    if (!DENSE) first[qi] = false;
                                    if (j == (DENSE ? n_list - 1 : last[qi])) tc_commit(&o_done[qi]);
                                    if (qi == lastq) tc_commit(&kv_empty[ST]);
                                }
                                if (more && visits(en, qi)) {
                                    if (!kv_ready) {
                                        const int gn = g + j + 1;
                                        if (!mbar_wait(&kv_full[ST ^ 1], (gn >> 1) & 1, p.status,
                                                       abort_flag))
                                            return false;
                                        tc_fence_after();
                                        kv_ready = true;
                                    }
                                    issue_s(qi, kst_next);
                                }
                            }
                            // every S product of the unit is issued: Q may be replaced
                            if (j + 2 == n_list) tc_commit(q_empty);
                            if (!DENSE) {
                                e = en;
                                en = enn;
                            }
                        }
                        return true;
                    };
                    const bool dense = ui->flags & 2;
                    if constexpr (kSolo) {
                        // One query tile (kSolo): key tile j's S/P sits in TMEM block j & 1,
                        // its K in K stage (g + j) % 3, its V in ring stage (g + j) & 1.
                        // S of tile j + 2 goes out right after P.V of tile j (in order on
                        // the tensor pipe, so it never overwrites a P still being read),
                        // while the softmax works on tile j + 1.
                        auto run_solo = [&]() -> bool {
                            auto issue_s_solo = [&](int j) -> bool {
                                const int t = g + j, ks = t % 3, sb = j & 1;
                                if (!mbar_wait(&k_full[ks], (t / 3) & 1, p.status, abort_flag))
                                    return false;
                                tc_fence_after();
                                const uint32_t kst = ks < 2 ? k_of(ks) : q_lo + (C::kQBytes >> 4);
#pragma unroll
                                for (int kk = 0; kk < D / 16; ++kk) {
                                    const uint32_t off = ((kk >> 2) * (kBM * 128) + (kk & 3) * 32) >> 4;
                                    tc_mma_ss(tmem + sb * kBN, desc_join(q_lo + off, dhi),
                                              desc_join(kst + off, dhi), idS, kk > 0 ? 1u : 0u);
                                }
                                tc_commit(&s_full[sb]);
                                tc_commit(&k_empty[ks]);
                                return true;
                            };
                            if (!issue_s_solo(0)) return false;
                            if (n_list > 1 && !issue_s_solo(1)) return false;
                            if (n_list <= 2) tc_commit(q_empty);
                            for (int j = 0; j < n_list; ++j) {
                                const int sb = j & 1, ST = (g + j) & 1;
                                // (the two P phase counters selected, not indexed: registers)
                                const uint32_t par = (sb ? pw[1] : pw[0]) & 1;
                                if (!mbar_wait(&p_full[sb], par, p.status, abort_flag))
                                    return false;
                                if (sb) ++pw[1]; else ++pw[0];
                                tc_fence_after();
                                if (j == 0 && uo[0] > 0) {
                                    // O still holds the previous unit until its epilogue
                                    // has read it
                                    if (!mbar_wait(&o_free[0], (uo[0] - 1) & 1, p.status, abort_flag))
                                        return false;
                                    tc_fence_after();
                                }
                                if (!mbar_wait(&kv_full[ST], ((g + j) >> 1) & 1, p.status, abort_flag))
                                    return false;
                                tc_fence_after();
                                const uint32_t vst = v_of(ST);
#pragma unroll
                                for (int kk = 0; kk < kBN / 16; ++kk)
                                    tc_mma_ts(tmem + 256, tmem + sb * kBN + kk * 8,
                                              desc_join(vst + ((kk * (16 * 128)) >> 4), dhi), idPV,
                                              (j > 0 || kk > 0) ? 1u : 0u);
                                tc_commit(pv_done);
                                if (j == n_list - 1) tc_commit(&o_done[0]);
                                tc_commit(&kv_empty[ST]);
                                if (j + 2 < n_list) {
                                    if (!issue_s_solo(j + 2)) return false;
                                    // every S product of the unit is issued: Q may be replaced
                                    if (j + 3 == n_list) tc_commit(q_empty);
                                }
                            }
                            return true;
                        };
                        if (ok) ok = run_solo();
                    } else if (ok) {
                        if (nq == 2)
                            ok = dense ? run(std::integral_constant<int, 2>{}, std::true_type{})
                                       : run(std::integral_constant<int, 2>{}, std::false_type{});
                        else
                            ok = dense ? run(std::integral_constant<int, 1>{}, std::true_type{})
                                       : run(std::integral_constant<int, 1>{}, std::false_type{});
                    }
                    for (int qi = 0; qi < 2; ++qi)
                        if ((dense && n_list > 0) ? qi < nq : last[qi] >= 0) ++uo[qi];
                    g += n_list;
                }
                if (ok) mbar_arrive(&unit_empty[slot]);
            }
            // every MMA issued by this thread has finished once this arrives
            tc_commit(mma_idle);
            mbar_drain(mma_idle, 0);
        }
    } else {
        // ------------------------------------------------------------ softmax
        const int qi = (warp - 2) >> 2;
        const int quarter = warp & 3;
        const int r = quarter * 32 + lane;
        const int qr = r >> pl2, hoff = r & ((1 << pl2) - 1);  // query row and head of tile row r
        const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
        const uint32_t tS = tmem + lane_base + qi * kBN;
        const uint32_t tO = tmem + lane_base + 256 + qi * 128;
        // Parities of the phases this warpgroup waits next, one bit each (all it
        // needs of its counters; one register across the key-tile loop):
        //   bit 0 / 1  metadata barrier of ring stage 0 / 1,
        //   bit 2      S barrier (kSolo: of S/P block 0),
        //   bit 3      O barrier (o_done),
        //   bit 4      ring stage of the unit's first key tile,
        //   bit 5      kSolo: S barrier of S/P block 1.
        uint32_t ph = 0;
        int npv = 0;  // kSolo: P.V products this warpgroup has handed P to so far
        bool ok = true;
        for (int k = 0; ok; ++k) {
            const int slot = k & 1;
            if (!mbar_wait(&unit_full[slot], (k >> 1) & 1, p.status, abort_flag)) break;
            const UnitInfo *ui = units + slot;
            if (ui->flags & 1) break;
            const int n_list = ui->n_list;
            const uint32_t st0 = (ph >> 4) & 1;  // stage of key tile 0 of this unit
            ph ^= (uint32_t)(n_list & 1) << 4;
            if (qi < ui->nq) {
                // (the unit's other fields are read again from its slot for the
                // epilogue: fewer registers live across the key-tile loop)
                const bool udense = ui->flags & 2;
                const int last = udense ? n_list - 1 : ui->last[qi];
                const int kklen = ui->kklen;
                // S_aug position of this thread's query row (-1: the tile row holds
                // no query row of the unit, and sees no key)
                int pos;
                if constexpr (kQC) {
                    // -1: the tile row holds no query row (it sees no key)
                    const int w = ui->qc[qi][r >> 5];
                    pos = lane < (w >> 24) ? (w & 0xffffff) + lane : -1;
                } else {
                    pos = ui->pbase + qi * (kPair ? 0 : ui->qstepu) + qr;
                }
                int rp = SONIC_ROLE_SYS, sp = 0;
                if (kQC ? pos >= 0 : pos <= ui->klen - 1) {
                    rp = p.role[ui->kstart + pos];
                    sp = p.seg[ui->kstart + pos];
                }
                const int32_t *lst = lists + slot * kMaxKTiles;
                // l: sum of the rounded probabilities (normalises O); l_lse: of the
                // unrounded ones, for the log-sum-exp output (kLse: lse requested)
                float m_used = -INFINITY, l = 0.f, l_lse = 0.f;
                // ln: the part of l on Nexus keys (kMass)
                float ln = 0.f;
                // the next list entry is read one tile ahead: shared memory is busy
                // feeding the tensor cores, so a load on the critical path is slow
                int entry = n_list > 0 ? lst[0] : 0;
                for (int j = 0; j <= last; ++j) {
                    const int e = entry;
                    entry = j + 1 < n_list ? lst[j + 1] : 0;
                    if (!udense && !((e >> (2 + qi)) & 1)) continue;  // a tile it does not see
                    const int st = (st0 + j) & 1;
                    const int kt = e >> 6;
                    const bool cut = (e >> qi) & 1;
                    const int nexus_keys = (e >> 4) & 3;
                    // The keys' masks are read on cut tiles only, their Nexus bits
                    // on tiles with some Nexus keys: one phase of this tile's
                    // metadata barrier each.
                    const bool need_meta = cut || (kMass && nexus_keys == 2);
                    if (need_meta) {
                        const uint32_t mph = (ph >> st) & 1;
                        ph ^= 1u << st;
                        if (!mbar_wait(&meta_full[2 * st + qi], mph, p.status, abort_flag)) {
                            ok = false;
                            break;
                        }
                    }
                    // The mask bits of a cut tile, worked out before S is read: the MMA
                    // producing S runs meanwhile, and the mask record and the S row are
                    // never held in registers together.
                    uint32_t mbits[4] = {0xffffffffu, 0xffffffffu, 0xffffffffu, 0xffffffffu};
                    if (cut) tile_mask_bits(tmasks + st, meta_role + st * kBN, meta_seg + st * kBN,
                                            meta_pos + st * kBN, pos, rp, sp, p.nexus_mode, mbits);
                    // kSolo: key tile j's S/P block and barriers are those of tile j & 1
                    // (parity bit 5 for block 1)
                    const int sb = kSolo ? (j & 1) : qi;
                    const uint32_t sbit = (kSolo && sb) ? 32u : 4u;
                    const uint32_t tSj = kSolo ? tS + (uint32_t)(sb * kBN) : tS;
                    if (!mbar_wait(&s_full[sb], (ph & sbit) ? 1u : 0u, p.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    ph ^= sbit;
                    tc_fence_after();
                    // S row into registers: four 32-column loads, one wait
                    uint32_t sr[4][32];
#pragma unroll
                    for (int c = 0; c < 4; ++c) tmem_ld32(tSj + c * 32, sr[c]);
                    tmem_ld_wait();
#pragma unroll
                    for (int c = 0; c < 4; ++c) reg_fence32(sr[c]);
                    // row maximum (masked keys set to -inf on a cut tile)
                    float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                    // 32-key chunks hidden from every row of the warp: no maximum, no
                    // exponentials, zero probabilities (bit c; warp-uniform)
                    uint32_t zchunk = 0;
                    if (!cut) {
#pragma unroll
                        for (int c = 0; c < 4; ++c)
#pragma unroll
                            for (int x = 0; x < 32; x += 2)
                                mx4[c] = fmax3(mx4[c], __uint_as_float(sr[c][x]),
                                               __uint_as_float(sr[c][x + 1]));
                    } else {
#pragma unroll
                        for (int c = 0; c < 4; ++c)
                        {
                            // chunks the whole warp sees, or sees none of, skip the
                            // per-key mask (both common away from a causal diagonal)
                            if (__all_sync(0xffffffffu, mbits[c] == 0xffffffffu)) {
#pragma unroll
                                for (int x = 0; x < 32; x += 2)
                                    mx4[c] = fmax3(mx4[c], __uint_as_float(sr[c][x]),
                                                   __uint_as_float(sr[c][x + 1]));
                            } else if (__all_sync(0xffffffffu, mbits[c] == 0u)) {
                                zchunk |= 1u << c;
                            } else {
#pragma unroll
                                for (int x = 0; x < 32; ++x) {
                                    if (!((mbits[c] >> x) & 1)) sr[c][x] = __float_as_uint(-INFINITY);
                                    mx4[c] = fmaxf(mx4[c], __uint_as_float(sr[c][x]));
                                }
                            }
                        }
                    }
                    const float mx =
                        fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3])) * p.scale_log2;
                    // (m_used = -inf: no visible key so far, so l = 0 and O = 0 --
                    // this tile starts the row whatever came before)
                    float alpha = 1.f, m_new = m_used;
                    if (m_used == -INFINITY) {
                        m_new = mx;
                    } else if (mx > m_used + kRescaleThreshold) {
                        m_new = mx;
                        alpha = ex2(m_used - m_new);
                    }
                    const float mref = (m_new == -INFINITY) ? 0.f : m_new;
                    // probabilities, written as bf16 pairs over the S columns
                    const float2 sc2 = make_float2(p.scale_log2, p.scale_log2);
                    const float2 nm2 = make_float2(-mref, -mref);
                    float ls[4] = {0.f, 0.f, 0.f, 0.f};
                    float2 rs2x = make_float2(0.f, 0.f);
                    // the Nexus part of the row sum: all of it, none, or (some Nexus
                    // keys) the keys the tile's Nexus bits select.  The two forms of
                    // the loop are separate instances, so the common one stays one
                    // straight run of code the compiler can interleave across chunks.
                    float lsn[2] = {0.f, 0.f};
                    auto exps = [&](auto nx_tag) {
                        constexpr bool NX = decltype(nx_tag)::value;
                        uint32_t nxb[4] = {0u, 0u, 0u, 0u};
                        if (NX) {
                            const uint4 nx = reinterpret_cast<const uint4 *>(tmasks + st)[1];
                            nxb[0] = nx.x;
                            nxb[1] = nx.y;
                            nxb[2] = nx.z;
                            nxb[3] = nx.w;
                        }
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            uint32_t pk[16];
                            if ((zchunk >> c) & 1) {
#pragma unroll
                                for (int x = 0; x < 16; ++x) pk[x] = 0u;
                                tmem_st16(tSj + c * 16, pk);
                                continue;
                            }
#pragma unroll
                            for (int x = 0; x < 32; x += 2) {
                                const float2 v = __ffma2_rn(make_float2(__uint_as_float(sr[c][x]),
                                                                        __uint_as_float(sr[c][x + 1])),
                                                            sc2, nm2);
                                const float2 eu = make_float2(ex2(v.x), ex2(v.y));
                                if (kLse) rs2x = __fadd2_rn(rs2x, eu);
                                const uint32_t pr = pack_bf16x2(eu.x, eu.y);
                                pk[x >> 1] = pr;
                                // the row sum adds the rounded probabilities P.V
                                // multiplies by, so O is a weighted mean of V rows with
                                // weights summing to one (rounding moves weight between
                                // keys, it does not scale the output)
                                add_bf16x2_to_f32(ls[(x >> 1) & 2], ls[((x >> 1) & 2) + 1], pr);
                                if (NX)
                                    add_bf16x2_to_f32_if(lsn[0], lsn[1], pr, nxb[c] & (1u << x),
                                                         nxb[c] & (2u << x));
                            }
                            tmem_st16(tSj + c * 16, pk);
                        }
                    };
                    if (kMass && nexus_keys == 2)
                        exps(std::true_type{});
                    else
                        exps(std::false_type{});
                    const float l_tile = (ls[0] + ls[1]) + (ls[2] + ls[3]);
                    l = l * alpha + l_tile;
                    if (kLse) l_lse = l_lse * alpha + (rs2x.x + rs2x.y);
                    if (kMass) ln = ln * alpha + (nexus_keys == 1 ? l_tile : (lsn[0] + lsn[1]));
                    // O rescale (the previous P.V of this tile is complete: this S
                    // was issued after it, and S is done)
                    if (__any_sync(0xffffffffu, alpha != 1.f)) {
                        if constexpr (kSolo) {
                            // the last P.V may still be accumulating into O: it is P.V
                            // number npv, and the one before it is done (this S was
                            // issued after it), so its phase is the one to wait for
                            if (!mbar_wait(pv_done, (npv - 1) & 1, p.status, abort_flag)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                        }
#pragma unroll
                        for (int c = 0; c < D / 32; ++c) {
                            uint32_t o[32];
                            tmem_ld32(tO + c * 32, o);
                            tmem_ld_wait();
                            reg_fence32(o);
#pragma unroll
                            for (int x = 0; x < 32; ++x)
                                o[x] = __float_as_uint(__uint_as_float(o[x]) * alpha);
                            tmem_st32(tO + c * 32, o);
                        }
                    }
                    tmem_st_wait();
                    // Rows of V past the sequence end: zero them so 0 * garbage
                    // cannot reach the accumulator (the warps of the first query
                    // tile visiting the key tile; its P.V is issued first).
                    const int first_qi = (udense || (e & 4)) ? 0 : 1;
                    if (qi == first_qi && kt * kBN + kBN > kklen && kt * kBN + r >= kklen) {
#pragma unroll
                        for (int hh = 0; hh < C::kHalves; ++hh) {
                            uint4 *vr = reinterpret_cast<uint4 *>(Vs + st * C::kKVBytes +
                                                                  hh * (kBN * 128) + r * 128);
#pragma unroll
                            for (int u = 0; u < 8; ++u) vr[u] = make_uint4(0, 0, 0, 0);
                        }
                        fence_proxy_async_smem();
                    }
                    tc_fence_before();
                    mbar_arrive(&p_full[sb]);
                    if (kSolo) ++npv;
                    m_used = m_new;
                }
                if (!ok) break;
                const int layer = ui->layer, h = ui->h0 + qi * (kPair ? 1 : ui->pairu) + hoff;
                // query row within the sequence
                const int qidx =
                    kQC ? pos - (ui->klen - ui->qlen)
                        : ui->qt * urows + qi * (kPair ? 0 : ui->qstepu) + qr;
                const bool row_ok = kQC ? pos >= 0 : pos <= ui->klen - 1 && qidx < ui->qlen;
                const int64_t qrow = (int64_t)ui->qstart + qidx;
                uint16_t *orow = p.O + layer * p.o_ls + (qrow * p.Hq + h) * D;
                const int64_t sidx = ((int64_t)layer * p.total_q_rows + qrow) * p.Hq + h;
                if (last >= 0) {
                    // ------------------------------------------------ epilogue
                    if (!mbar_wait(&o_done[qi], (ph >> 3) & 1, p.status, abort_flag)) break;
                    ph ^= 8u;
                    tc_fence_after();
                    const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t o[32];
                        tmem_ld32(tO + c * 32, o);
                        tmem_ld_wait();
                        reg_fence32(o);
                        if (c == D / 32 - 1) {
                            // O is read: the next unit's first P.V may overwrite it
                            tc_fence_before();
                            mbar_arrive(&o_free[qi]);
                        }
                        if (row_ok) {
                            // a thread writes its own row: in 32-byte stores a warp's
                            // store fills 32 whole L2 sectors, in 16-byte ones half of each
                            uint32_t w[16];
#pragma unroll
                            for (int x = 0; x < 16; ++x)
                                w[x] = pack_bf16x2(__uint_as_float(o[2 * x]) * inv,
                                                   __uint_as_float(o[2 * x + 1]) * inv);
                            if (p.o_v8) {
                                st_global_v8(orow + c * 32, w);
                                st_global_v8(orow + c * 32 + 16, w + 8);
                            } else {
                                uint4 *dst = reinterpret_cast<uint4 *>(orow + c * 32);
#pragma unroll
                                for (int u = 0; u < 4; ++u)
                                    dst[u] = make_uint4(w[4 * u], w[4 * u + 1], w[4 * u + 2], w[4 * u + 3]);
                            }
                        }
                    }
                    if (row_ok) {
                        if (kLse)
                            p.lse[sidx] = l_lse > 0.f ? (m_used + __log2f(l_lse)) * kLn2f : -INFINITY;
                        if (kMass) p.nexus_mass[sidx] = ln * inv;
                    }
                } else if (row_ok) {
                    // no key tile to visit (never for a valid layout): zeros
                    uint4 *dst = reinterpret_cast<uint4 *>(orow);
#pragma unroll
                    for (int u = 0; u < D / 8; ++u) dst[u] = make_uint4(0, 0, 0, 0);
                    if (kLse) p.lse[sidx] = -INFINITY;
                    if (kMass) p.nexus_mass[sidx] = 0.f;
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&unit_empty[slot]);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // After an abort no thread waits any more; let the copies the producer
    // issued land before the block's shared memory goes away.
    if (*abort_flag && warp == 0 && lane == 0) {
        if (issued_q > 0) mbar_drain(q_full, (issued_q - 1) & 1);
        for (int u = max(0, issued_kv - 2); u < issued_kv; ++u)
            mbar_drain(&kv_full[u & 1], (u >> 1) & 1);
        if (kSolo)
            for (int u = max(0, issued_k - 3); u < issued_k; ++u)
                mbar_drain(&k_full[u % 3], (u / 3) & 1);
    }
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------- key order
// Retained-first order.  Sequence b's keys are rewritten into rows
// [key_start[b], key_start[b] + span_b) of the workspace, span_b =
// align128(k_len[b]) + 128: first its retained keys (every role but body, in
// S_aug order), padded to a 128-row boundary, then its body keys (S_aug
// order), then padding to the end of the span.  Padding rows have role 255,
// position INT_MAX and source -1 (their K/V rows are zeroed).  key_start has
// B + 1 entries; the last is the number of rows written (every one of them
// gets a source index, so the copy kernel reads no unwritten entry).
constexpr int kOrderThreads = 1024;

__device__ __forceinline__ int span_of(int len) { return (len + kBN - 1) / kBN * kBN + kBN; }


__global__ void __launch_bounds__(kOrderThreads)
key_order_kernel(const uint8_t *__restrict__ role, const int32_t *__restrict__ seg,
                 const int32_t *__restrict__ k_start, const int32_t *__restrict__ k_len,
                 const int32_t *__restrict__ q_len, int B,
                 int max_k_len, int64_t total_rows, int64_t capacity,
                 int32_t *__restrict__ key_start,
                 int32_t *__restrict__ key_len, uint8_t *__restrict__ o_role,
                 int32_t *__restrict__ o_seg, int32_t *__restrict__ o_pos,
                 int32_t *__restrict__ o_src, int32_t *__restrict__ direct, int max_k_tiles,
                 int32_t *__restrict__ status) {
    const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    __shared__ int sh[2][32];
    __shared__ long long sh_base;
    __shared__ int sh_r, sh_smin, sh_first;
    // start of this sequence's span: the spans of the sequences before it
    long long base = 0;
    for (int i = tid; i < b; i += kOrderThreads)
        base += span_of(seq_rows(k_start[i], k_len[i], max_k_len, total_rows));
    if (tid == 0) {
        sh_base = 0;
        sh_r = 0;
        sh_smin = INT_MAX;
        sh_first = INT_MAX;
    }
    __syncthreads();
    if (base) atomicAdd(reinterpret_cast<unsigned long long *>(&sh_base), (unsigned long long)base);
    const int len_in = k_len[b];
    const int ks = k_start[b];
    const int len = seq_rows(ks, len_in, max_k_len, total_rows);
    if (tid == 0 && len != len_in) set_status(status, SONIC_ERR_INVALID_ARGUMENT);
    int cnt = 0;
    for (int i = tid; i < len; i += kOrderThreads) cnt += role[ks + i] != SONIC_ROLE_BODY;
    cnt = __reduce_add_sync(0xffffffffu, cnt);
    if (lane == 0 && cnt) atomicAdd(&sh_r, cnt);
    // the smallest segment among the query rows (the last q_len rows): a body
    // row of an earlier segment is seen by no query row of this call
    const int ql = min(max(q_len[b], 0), len);
    int smin = INT_MAX;
    for (int i = len - ql + tid; i < len; i += kOrderThreads) smin = min(smin, seg[ks + i]);
    smin = __reduce_min_sync(0xffffffffu, smin);
    if (lane == 0 && smin != INT_MAX) atomicMin(&sh_smin, smin);
    __syncthreads();
    const int s_min = sh_smin;
    const long long start = sh_base;
    const int R = sh_r, span = span_of(len);
    if (b == B - 1 && tid == 0) key_start[B] = (int32_t)min(start + span, (long long)capacity);
    if (start + span > capacity) {
        // the spans overflow the workspace (sequences that share key rows can
        // sum to more than total_k_rows): this sequence gets no keys, and the
        // rows of its span that exist become padding
        for (long long i = start + tid; i < capacity; i += kOrderThreads) {
            o_role[i] = 255;
            o_seg[i] = 0;
            o_pos[i] = INT_MAX;
            o_src[i] = -1;
        }
        if (tid == 0) {
            set_status(status, SONIC_ERR_WORKSPACE);
            key_start[b] = 0;
            key_len[b] = 0;
        }
        return;
    }
    const int body0 = (R + kBN - 1) / kBN * kBN;
    int kept = 0, bodies = 0;
    for (int c0 = 0; c0 < len; c0 += kOrderThreads) {
        const int i = c0 + tid;
        const bool valid = i < len;
        const int r = valid ? role[ks + i] : SONIC_ROLE_BODY;
        const bool keep = valid && r != SONIC_ROLE_BODY, body = valid && r == SONIC_ROLE_BODY;
        const unsigned bk = __ballot_sync(0xffffffffu, keep), bb = __ballot_sync(0xffffffffu, body);
        if (lane == 0) {
            sh[0][warp] = __popc(bk);
            sh[1][warp] = __popc(bb);
        }
        __syncthreads();
        int pk = 0, pb = 0, tk = 0, tb = 0;
        for (int w = 0; w < kOrderThreads / 32; ++w) {
            if (w < warp) {
                pk += sh[0][w];
                pb += sh[1][w];
            }
            tk += sh[0][w];
            tb += sh[1][w];
        }
        const unsigned below = (1u << lane) - 1u;
        if (valid) {
            const int dst = keep ? kept + pk + __popc(bk & below) : body0 + bodies + pb + __popc(bb & below);
            const int64_t o = start + dst;
            const int sv = seg[ks + i];
            o_role[o] = (uint8_t)r;
            o_seg[o] = sv;
            o_pos[o] = i;
            o_src[o] = ks + i;
            if (body && sv >= s_min) atomicMin(&sh_first, dst - body0);
        }
        kept += tk;
        bodies += tb;
        __syncthreads();
    }
    // padding: between the retained keys and the bodies, and after the bodies
    const int lp = body0 + (len - R);
    for (int i = tid; i < span; i += kOrderThreads) {
        if ((i >= R && i < body0) || i >= lp) {
            o_role[start + i] = 255;
            o_seg[start + i] = 0;
            o_pos[start + i] = INT_MAX;
            o_src[start + i] = -1;
        }
    }
    // Whole 128-row tiles of bodies before the first body row a query row can
    // see are never visited: their K/V rows are not copied (src -2).  A tile
    // holding any such row is copied whole, so a masked key never carries
    // stale data into P.V.
    __syncthreads();
    const int first = min(sh_first, len - R);  // body rows before it: unseen
    for (int i = body0 + tid; i < body0 + (first / kBN) * kBN; i += kOrderThreads)
        o_src[start + i] = -2;
    // A tile whose 128 rows are 128 consecutive rows of the input (a run of one
    // body, of the system prompt, of the current turn) is read by the attention
    // kernel from K and V themselves: it is not copied (source -2) and its first
    // input row is recorded; every other tile records -1 and is copied.
    __syncthreads();
    const int n_tiles = span / kBN;
    for (int t = warp; t < max_k_tiles; t += kOrderThreads / 32) {
        int d = -1;
        if (t < n_tiles) {
            const int64_t r0 = start + (int64_t)t * kBN;
            const int32_t s0 = o_src[r0];
            bool run = s0 >= 0;
#pragma unroll
            for (int w = 0; w < 4; ++w) run = run && o_src[r0 + w * 32 + lane] == s0 + w * 32 + lane;
            if (__all_sync(0xffffffffu, run)) {
                d = s0;
#pragma unroll
                for (int w = 0; w < 4; ++w) o_src[r0 + w * 32 + lane] = -2;
            }
        }
        if (lane == 0) direct[(int64_t)b * max_k_tiles + t] = d;
    }
    if (tid == 0) {
        key_start[b] = (int32_t)start;
        key_len[b] = lp;
    }
}

// ---------------------------------------------------------------- query order
// Retained-first query order.  A sequence's query rows (its last q_len rows)
// are walked as [body rows | every other row], each part in S_aug order and
// cut into runs: consecutive rows of one body, or consecutive rows that are
// not body rows.  Each run starts on a 32-row boundary and the second part on
// a 128-row boundary, so a 128-row query tile is four 32-row chunks, each
// chunk a stretch of at most 32 consecutive query rows of one run, and the
// rows of one body fill whole tiles of their own (the rows a body row sees are
// the same for its whole segment; in the given order a tile straddles two
// segments and the Nexus rows between them).  The chunk table holds, per
// sequence, chunks_per_seq words: (rows << 24) | first query row, 0 for a
// chunk without rows.  A sequence with more than kQRunsMax runs, or whose runs
// need more than align128(q_len) + kQSlack rows, keeps the given order (chunks
// of 32 consecutive query rows).
constexpr int kQOrderThreads = 1024;
constexpr int kQRunsMax = 1024;
constexpr int kQSlack = 1024;

// Exclusive prefix sum over the block (kQOrderThreads threads) and the total.
__device__ __forceinline__ int block_excl_scan(int v, int *sh, int &total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) sh[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = sh[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        sh[lane] = w;
    }
    __syncthreads();
    total = sh[31];
    const int r = x - v + (warp > 0 ? sh[warp - 1] : 0);
    __syncthreads();
    return r;
}

__global__ void __launch_bounds__(kQOrderThreads)
query_order_kernel(const uint8_t *__restrict__ role, const int32_t *__restrict__ seg,
                   const int32_t *__restrict__ k_start, const int32_t *__restrict__ k_len,
                   const int32_t *__restrict__ q_len, int max_k_len, int64_t total_rows,
                   int chunks_per_seq, int32_t *__restrict__ qchunks) {
    const int b = blockIdx.x, tid = threadIdx.x;
    __shared__ int sh[32];
    __shared__ int rs[kQRunsMax + 1];   // first query row of each run
    __shared__ int vs[kQRunsMax + 1];   // runs sorted by their place: first chunk row
    __shared__ int ss[kQRunsMax];       // ... first query row
    __shared__ int ls[kQRunsMax];       // ... rows
    const int ks = k_start[b];
    const int len = seq_rows(ks, k_len[b], max_k_len, total_rows);
    // a sequence the attention kernel refuses gets the given order; nothing
    // of it is read here beyond its rows
    const int ql = min(max(q_len[b], 0), len);
    const int q0 = ks + len - ql;  // row of query 0
    int32_t *out = qchunks + (int64_t)b * chunks_per_seq;
    // runs: their first rows in order
    int nr = 0;
    for (int c0 = 0; c0 < ql; c0 += kQOrderThreads) {
        const int i = c0 + tid;
        bool start = false;
        if (i < ql) {
            const bool body = role[q0 + i] == SONIC_ROLE_BODY;
            if (i == 0) {
                start = true;
            } else {
                const bool pbody = role[q0 + i - 1] == SONIC_ROLE_BODY;
                start = body != pbody || (body && seg[q0 + i] != seg[q0 + i - 1]);
            }
        }
        int total;
        const int at = block_excl_scan(start ? 1 : 0, sh, total);
        if (start && nr + at < kQRunsMax) rs[nr + at] = i;
        nr += total;
    }
    const bool many = nr > kQRunsMax;
    if (tid == 0 && !many) rs[nr] = ql;
    __syncthreads();
    // each run's place: body runs first, in order, then the other runs
    int rows = 0, isb = 0;
    if (!many && tid < nr) {
        rows = rs[tid + 1] - rs[tid];
        isb = role[q0 + rs[tid]] == SONIC_ROLE_BODY;
    }
    const int a32 = (rows + 31) & ~31;
    int tb, tn, nb_runs, n_other;
    const int eb = block_excl_scan(isb ? a32 : 0, sh, tb);
    const int en = block_excl_scan(isb ? 0 : a32, sh, tn);
    const int rb = block_excl_scan(isb ? 1 : 0, sh, nb_runs);
    const int ro = block_excl_scan((!many && tid < nr && !isb) ? 1 : 0, sh, n_other);
    const int other0 = (tb + 127) & ~127;
    const int span = other0 + tn;
    const bool given = many || span > ((ql + 127) & ~127) + kQSlack;
    if (!given && tid < nr) {
        const int k = isb ? rb : nb_runs + ro;
        vs[k] = isb ? eb : other0 + en;
        ss[k] = rs[tid];
        ls[k] = rows;
    }
    if (tid == 0 && !given) vs[nr] = INT_MAX;
    __syncthreads();
    for (int c = tid; c < chunks_per_seq; c += kQOrderThreads) {
        int w = 0;
        const int v = c * 32;
        if (given) {
            if (v < ql) w = (min(32, ql - v) << 24) | v;
        } else if (v < span) {
            // the last run placed at or before row v
            int lo = 0, hi = nr - 1;
            while (lo < hi) {
                const int mid = (lo + hi + 1) >> 1;
                if (vs[mid] <= v) lo = mid; else hi = mid - 1;
            }
            const int off = v - vs[lo];
            if (off >= 0 && off < ls[lo]) w = (min(32, ls[lo] - off) << 24) | (ss[lo] + off);
        }
        out[c] = w;
    }
}

// K and V rows of every layer into the retained-first order (warp per row;
// rows with source -1 are zeroed).
constexpr int kPermThreads = 256;

__device__ __forceinline__ int4 ld_nc(const void *ptr) {
    int4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.s32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(ptr));
    return v;
}

__global__ void __launch_bounds__(kPermThreads)
kv_permute_kernel(const uint8_t *__restrict__ K, const uint8_t *__restrict__ V,
                  uint8_t *__restrict__ Kp, uint8_t *__restrict__ Vp,
                  const int32_t *__restrict__ src, const int32_t *__restrict__ key_start, int B,
                  int64_t row_bytes, int64_t in_layer_bytes, int64_t out_layer_bytes) {
    const int layer = blockIdx.y >> 1;
    const bool is_v = blockIdx.y & 1;
    const uint8_t *in = (is_v ? V : K) + (int64_t)layer * in_layer_bytes;
    uint8_t *out = (is_v ? Vp : Kp) + (int64_t)layer * out_layer_bytes;
    const int64_t n_rows = key_start[B];
    const int lane = threadIdx.x & 31;
    const int64_t n_warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int cpr = (int)(row_bytes >> 4);
    for (int64_t r = (((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5); r < n_rows;
         r += n_warps) {
        const int32_t s = src[r];
        if (s == -2) continue;  // a body tile no query row of the call sees
        const uint8_t *pi = in + (int64_t)s * row_bytes;
        uint8_t *po = out + r * row_bytes;
        for (int c0 = lane; c0 < cpr; c0 += 32 * 4) {
            int4 v[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int c = c0 + 32 * u;
                v[u] = make_int4(0, 0, 0, 0);
                if (c < cpr && s >= 0) v[u] = ld_nc(pi + ((int64_t)c << 4));
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int c = c0 + 32 * u;
                if (c < cpr) *reinterpret_cast<int4 *>(po + ((int64_t)c << 4)) = v[u];
            }
        }
    }
}

template <int D>
cudaError_t launch_prefill(const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv,
                           const CUtensorMap &tk0, const CUtensorMap &tv0, const CUtensorMap &tq32,
                           const PfParams &p, bool solo, int grid, cudaStream_t s) {
    constexpr size_t smem = PfCfg<D>::kSmem;
    static_assert(smem <= 232448, "prefill shared memory");
    const int out = (p.lse != nullptr ? 1 : 0) | (p.nexus_mass != nullptr ? 2 : 0);
    // instances: chunked query order (paired or not), single-tile units, or the
    // given order (paired or not)
    using K = void (*)(CUtensorMap, CUtensorMap, CUtensorMap, CUtensorMap, CUtensorMap,
                       CUtensorMap, PfParams);
    auto pick = [&](auto qc, auto solo_t, auto pair_t) -> K {
        constexpr bool a = decltype(qc)::value, b = decltype(solo_t)::value,
                       c = decltype(pair_t)::value;
        return out == 0   ? (K)prefill_kernel<D, 0, a, b, c>
               : out == 1 ? (K)prefill_kernel<D, 1, a, b, c>
               : out == 2 ? (K)prefill_kernel<D, 2, a, b, c>
                          : (K)prefill_kernel<D, 3, a, b, c>;
    };
    using T = std::true_type;
    using F = std::false_type;
    const bool paired = p.pair != 0;
    K kern = p.qchunks != nullptr ? (paired ? pick(T{}, F{}, T{}) : pick(T{}, F{}, F{}))
             : solo               ? pick(F{}, T{}, F{})
             : paired             ? pick(F{}, F{}, T{})
                                  : pick(F{}, F{}, F{});
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, kPfThreads, smem, s>>>(tq, tk, tv, tk0, tv0, tq32, p);
    return cudaGetLastError();
}

// Chunk words per sequence of the retained-first query order: room for
// align128(max_q_len) + kQSlack query-tile rows.
int query_chunks_of(const sonic_prefill_args *a) {
    return ((a->max_q_len + kBM - 1) / kBM * kBM + kQSlack) / 32;
}

int max_k_tiles_of(const sonic_prefill_args *a) {
    const int t = (a->max_k_len + kBN - 1) / kBN;
    return a->key_order == SONIC_KEYS_RETAINED_FIRST ? t + 1 : t;
}

// Workspace: the work-unit counter, tile summaries and tile column masks; with
// the retained-first order also the permuted key metadata and the permuted K
// and V of every layer.
struct PfWorkspace {
    size_t counter, sums, masks, key_start, key_len, role, seg, pos, src, direct, qchunks, kp, vp,
        total;
    int64_t rows;  // rows of the permuted K/V per layer
};

PfWorkspace workspace_layout(const sonic_prefill_args *a) {
    PfWorkspace w{};
    const size_t tiles = (size_t)a->batch * max_k_tiles_of(a);
    w.counter = 0;
    w.sums = 256;
    w.masks = w.sums + round_up(tiles * sizeof(TileSum), 256);
    size_t off = w.masks + round_up(tiles * sizeof(TileMasks), 256);
    if (a->key_order == SONIC_KEYS_RETAINED_FIRST) {
        const int64_t span = (int64_t)((a->max_k_len + kBN - 1) / kBN) * kBN + kBN;
        w.rows = std::min<int64_t>((int64_t)a->batch * span,
                                   (int64_t)a->total_k_rows + (int64_t)2 * kBN * a->batch);
        auto take = [&](size_t bytes) {
            const size_t o = off;
            off += round_up(bytes, 256);
            return o;
        };
        w.key_start = take((size_t)(a->batch + 1) * 4);
        w.key_len = take((size_t)a->batch * 4);
        w.role = take((size_t)w.rows);
        w.seg = take((size_t)w.rows * 4);
        w.pos = take((size_t)w.rows * 4);
        w.src = take((size_t)w.rows * 4);
        w.direct = take(tiles * 4);
        w.qchunks = take((size_t)a->batch * query_chunks_of(a) * 4);
        const size_t layer = (size_t)w.rows * a->n_heads_kv * a->head_dim * 2;
        w.kp = take(layer * a->n_layers);
        w.vp = take(layer * a->n_layers);
    }
    w.total = off;
    return w;
}

}  // namespace
}  // namespace sonic

using namespace sonic;

extern "C" size_t sonic_prefill_workspace_size(const sonic_prefill_args *a) {
    if (a == nullptr || a->batch <= 0 || a->max_k_len <= 0) return 0;
    if (a->key_order == SONIC_KEYS_RETAINED_FIRST &&
        (a->n_layers < 1 || a->n_heads_kv < 1 || a->head_dim < 1 || a->total_k_rows < 0))
        return 0;
    return workspace_layout(a).total;
}

extern "C" sonic_status_t sonic_attn_prefill(const uint16_t *Q, const uint16_t *K,
                                             const uint16_t *V, const int32_t *seg_id,
                                             const uint8_t *role, uint16_t *O,
                                             const sonic_prefill_args *a,
                                             sonic_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (a == nullptr) return SONIC_ERR_INVALID_ARGUMENT;
    if (a->batch < 0 || a->n_layers < 1 || a->n_heads_kv < 1 || a->n_heads_q < 1 ||
        a->n_heads_q % a->n_heads_kv != 0 || a->max_q_len < 0 || a->max_k_len < 0 ||
        a->total_q_rows < 0 || a->total_k_rows < 0)
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->batch == 0 || a->max_q_len == 0) return SONIC_OK;
    if (Q == nullptr || K == nullptr || V == nullptr || O == nullptr || role == nullptr ||
        seg_id == nullptr || a->k_start == nullptr || a->k_len == nullptr ||
        a->q_start == nullptr || a->q_len == nullptr)
        return SONIC_ERR_INVALID_ARGUMENT;
    const int D = a->head_dim;
    if (D != 64 && D != 128) return SONIC_ERR_UNSUPPORTED;
    if (a->nexus_vis != SONIC_NEXUS_FULL && a->nexus_vis != SONIC_NEXUS_CAUSAL_SEGMENTS)
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->key_order != SONIC_KEYS_AS_GIVEN && a->key_order != SONIC_KEYS_RETAINED_FIRST)
        return SONIC_ERR_INVALID_ARGUMENT;
    const bool reorder = a->key_order == SONIC_KEYS_RETAINED_FIRST;
    if (a->max_k_len < a->max_q_len || a->total_k_rows == 0 || a->total_q_rows == 0)
        return SONIC_ERR_INVALID_ARGUMENT;
    if (max_k_tiles_of(a) > kMaxKTiles) return SONIC_ERR_UNSUPPORTED;
    if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O))
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->n_layers > 1 && (a->q_layer_stride <= 0 || a->kv_layer_stride <= 0 ||
                            a->o_layer_stride <= 0 || (a->q_layer_stride * 2) % 16 != 0 ||
                            (a->kv_layer_stride * 2) % 16 != 0 ||
                            (a->o_layer_stride * 2) % 16 != 0))
        return SONIC_ERR_INVALID_ARGUMENT;
    const size_t need = sonic_prefill_workspace_size(a);
    if (a->workspace == nullptr || a->workspace_bytes < need) return SONIC_ERR_WORKSPACE;
    if (reorder && workspace_layout(a).rows > (int64_t)0x7fffffff - kBN)
        return SONIC_ERR_UNSUPPORTED;
    // Query heads packed per tile (a power of two dividing G): short query
    // blocks take 256 / P rows per block instead of leaving tile rows empty.
    const int G = a->n_heads_q / a->n_heads_kv;
    int pack_log2 = 0;
    while ((G % (2 << pack_log2)) == 0 && pack_log2 < 3 &&
           (long long)a->max_q_len * (2 << pack_log2) <= 2 * kBM)
        ++pack_log2;
    const int R = kBM >> pack_log2;
    // Unpacked heads in pairs sharing a KV head: a unit's two query tiles
    // then see the same keys (no key tile visited by one tile alone).
    const bool pair = pack_log2 == 0 && G % 2 == 0;
    const long long urows = pair ? R : 2 * R;
    // retained-first keys with unpacked heads: the query rows are walked in
    // the retained-first order too, as 32-row chunks (query_order_kernel)
    const bool qchunked = reorder && pack_log2 == 0;
    const long long qrows_v = qchunked ? (long long)query_chunks_of(a) * 32 : a->max_q_len;
    const long long qtiles = (qrows_v + urows - 1) / urows;
    const long long HG = pair ? a->n_heads_q / 2 : a->n_heads_q >> pack_log2;
    const long long n_units = qtiles * HG * a->batch * a->n_layers;
    if (n_units > 0x7fffffff) return SONIC_ERR_UNSUPPORTED;

    const uint64_t qrow = (uint64_t)a->n_heads_q * D, krow = (uint64_t)a->n_heads_kv * D;
    const uint64_t q_layer = a->n_layers > 1 ? (uint64_t)a->q_layer_stride * 2
                                             : (uint64_t)a->total_q_rows * qrow * 2;
    const uint64_t k_layer = a->n_layers > 1 ? (uint64_t)a->kv_layer_stride * 2
                                             : (uint64_t)a->total_k_rows * krow * 2;
    const uint64_t qd[4] = {(uint64_t)D, (uint64_t)a->n_heads_q, (uint64_t)a->total_q_rows,
                            (uint64_t)a->n_layers};
    const uint64_t qs[3] = {(uint64_t)D * 2, qrow * 2, q_layer};
    const PfWorkspace ws = workspace_layout(a);
    uint8_t *wsb = static_cast<uint8_t *>(a->workspace);
    // K/V rows the tiles are cut from: the inputs, or their permuted copies
    const void *Kt = reorder ? (const void *)(wsb + ws.kp) : (const void *)K;
    const void *Vt = reorder ? (const void *)(wsb + ws.vp) : (const void *)V;
    const uint64_t kt_rows = reorder ? (uint64_t)ws.rows : (uint64_t)a->total_k_rows;
    const uint64_t kt_layer = reorder ? (uint64_t)ws.rows * krow * 2 : k_layer;
    // Whole Q, K and V tiles: 5-D maps (64 columns, head, row, 64-column half,
    // layer), so one copy brings both halves of a head_dim-128 tile, each half a
    // [row][128-byte] block as the 128-byte swizzle wants it.
    const uint64_t nh = (uint64_t)D / 64;
    const uint64_t qd5[5] = {64, (uint64_t)a->n_heads_q, (uint64_t)a->total_q_rows, nh,
                             (uint64_t)a->n_layers};
    const uint64_t qs5[4] = {(uint64_t)D * 2, qrow * 2, 128, q_layer};
    const uint32_t qbox5[5] = {64, 1u << pack_log2, (uint32_t)R, (uint32_t)nh, 1};  // R rows x P heads
    const uint64_t kd5[5] = {64, (uint64_t)a->n_heads_kv, kt_rows, nh, (uint64_t)a->n_layers};
    const uint64_t ks5[4] = {(uint64_t)D * 2, krow * 2, 128, kt_layer};
    const uint32_t box5[5] = {64, 1, 128, (uint32_t)nh, 1};
    CUtensorMap tq, tk, tv, tk0, tv0, tq32;
    if (!make_tmap_bf16_5d(&tq, Q, qd5, qs5, qbox5) || !make_tmap_bf16_5d(&tk, Kt, kd5, ks5, box5) ||
        !make_tmap_bf16_5d(&tv, Vt, kd5, ks5, box5))
        return SONIC_ERR_INVALID_ARGUMENT;
    // the inputs themselves, for the retained-first tiles read in place
    const uint64_t kd0[5] = {64, (uint64_t)a->n_heads_kv, (uint64_t)a->total_k_rows, nh,
                             (uint64_t)a->n_layers};
    const uint64_t ks0[4] = {(uint64_t)D * 2, krow * 2, 128, k_layer};
    if (reorder) {
        if (!make_tmap_bf16_5d(&tk0, K, kd0, ks0, box5) ||
            !make_tmap_bf16_5d(&tv0, V, kd0, ks0, box5))
            return SONIC_ERR_INVALID_ARGUMENT;
    } else {
        tk0 = tk;
        tv0 = tv;
    }
    const uint32_t qbox32[4] = {64, 1, 32, 1};  // one 32-row query chunk of one head
    if (qchunked) {
        if (!make_tmap_bf16_4d(&tq32, Q, qd, qs, qbox32)) return SONIC_ERR_INVALID_ARGUMENT;
    } else {
        tq32 = tq;
    }

    PfParams p{};
    p.k_start = a->k_start;
    p.k_len = a->k_len;
    p.q_start = a->q_start;
    p.q_len = a->q_len;
    p.role = role;
    p.seg = seg_id;
    p.key_start = a->k_start;
    p.key_len = a->k_len;
    p.key_role = role;
    p.key_seg = seg_id;
    p.key_pos = nullptr;
    p.key_direct = nullptr;
    p.qchunks = nullptr;
    p.qchunks_per_seq = 0;
    if (qchunked) {
        p.qchunks = reinterpret_cast<const int32_t *>(wsb + ws.qchunks);
        p.qchunks_per_seq = query_chunks_of(a);
    }
    if (reorder) {
        p.key_start = reinterpret_cast<const int32_t *>(wsb + ws.key_start);
        p.key_len = reinterpret_cast<const int32_t *>(wsb + ws.key_len);
        p.key_role = wsb + ws.role;
        p.key_seg = reinterpret_cast<const int32_t *>(wsb + ws.seg);
        p.key_pos = reinterpret_cast<const int32_t *>(wsb + ws.pos);
        p.key_direct = reinterpret_cast<const int32_t *>(wsb + ws.direct);
    }
    p.O = O;
    p.lse = a->lse;
    p.nexus_mass = a->nexus_mass;
    p.status = a->status;
    p.sums = reinterpret_cast<const TileSum *>(wsb + ws.sums);
    p.masks = reinterpret_cast<const TileMasks *>(wsb + ws.masks);
    p.counter = reinterpret_cast<int32_t *>(wsb + ws.counter);
    p.n_units = (int)n_units;
    p.qtiles = (int)qtiles;
    p.HG = (int)HG;
    p.max_k_tiles = max_k_tiles_of(a);
    p.max_k_len = a->max_k_len;
    p.B = a->batch;
    p.Hq = a->n_heads_q;
    p.G = G;
    p.total_k_rows = a->total_k_rows;
    p.pack_log2 = pack_log2;
    p.pair = pair ? 1 : 0;
    p.o_ls = a->o_layer_stride;
    p.o_v8 = (reinterpret_cast<uintptr_t>(O) % 32 == 0) && (a->o_layer_stride * 2) % 32 == 0;
    p.total_q_rows = a->total_q_rows;
    const float scale = a->softmax_scale > 0.f ? a->softmax_scale : 1.0f / sqrtf((float)D);
    p.scale_log2 = scale * kLog2ef;
    p.nexus_mode = a->nexus_vis;

    if (reorder) {
        key_order_kernel<<<a->batch, kOrderThreads, 0, stream>>>(
            role, seg_id, a->k_start, a->k_len, a->q_len, a->batch, a->max_k_len, a->total_k_rows,
            ws.rows,
            reinterpret_cast<int32_t *>(wsb + ws.key_start),
            reinterpret_cast<int32_t *>(wsb + ws.key_len), wsb + ws.role,
            reinterpret_cast<int32_t *>(wsb + ws.seg), reinterpret_cast<int32_t *>(wsb + ws.pos),
            reinterpret_cast<int32_t *>(wsb + ws.src), reinterpret_cast<int32_t *>(wsb + ws.direct),
            max_k_tiles_of(a), a->status);
        const int sms = device_sm_count();
        // ~32 blocks per SM in all, as in the compaction copy
        const int per_slice = std::max(1, (sms * 32 + 2 * a->n_layers - 1) / (2 * a->n_layers));
        kv_permute_kernel<<<dim3(per_slice, 2 * a->n_layers), kPermThreads, 0, stream>>>(
            reinterpret_cast<const uint8_t *>(K), reinterpret_cast<const uint8_t *>(V),
            wsb + ws.kp, wsb + ws.vp, reinterpret_cast<const int32_t *>(wsb + ws.src),
            reinterpret_cast<const int32_t *>(wsb + ws.key_start), a->batch, (int64_t)krow * 2,
            (int64_t)k_layer, (int64_t)kt_layer);
    }
    if (qchunked)
        query_order_kernel<<<a->batch, kQOrderThreads, 0, stream>>>(
            role, seg_id, a->k_start, a->k_len, a->q_len, a->max_k_len, a->total_k_rows,
            p.qchunks_per_seq, reinterpret_cast<int32_t *>(wsb + ws.qchunks));
    tile_summary_kernel<<<dim3(p.max_k_tiles, a->batch), 128, 0, stream>>>(
        p.key_role, p.key_seg, p.key_pos, p.key_start, p.key_len,
        reinterpret_cast<TileSum *>(wsb + ws.sums), reinterpret_cast<TileMasks *>(wsb + ws.masks),
        p.max_k_tiles,
        reorder ? (int64_t)ws.rows : (int64_t)a->total_k_rows, a->status, p.counter);
    // one persistent block per SM (fewer when there are fewer units)
    const int grid = (int)std::min<long long>(device_sm_count(), n_units);
    // every unit holds one query tile: packed heads with every query block within
    // one tile (R rows), so the second tile's TMEM block and Q buffer are free
    const bool solo = !qchunked && pack_log2 > 0 && a->max_q_len <= R;
    cudaError_t e = (D == 128)
                        ? launch_prefill<128>(tq, tk, tv, tk0, tv0, tq32, p, solo, grid, stream)
                        : launch_prefill<64>(tq, tk, tv, tk0, tv0, tq32, p, solo, grid, stream);
    return e == cudaSuccess ? SONIC_OK : SONIC_ERR_CUDA;
}
