// GQA decode over the retained (compacted) KV cache.
//
// One generation step (SONIC App. C: generation conditions on I_sys, the
// Nexus state and the current query, i.e. on exactly the rows compaction
// kept).  Every retained row of a sequence is visible to its new token.
//
// Split-K, HBM-bound design:
//   decode_tc      persistent blocks (one per SM) claim units (key chunk, KV
//                  head, sequence, layer) from a counter and stream their K/V
//                  tiles of 128 keys through a TMA ring; both contractions run
//                  on the tensor cores with the keys in the M dimension (see
//                  the kernel's comment); a single-chunk sequence writes O
//                  directly, otherwise the partial (max, sum, unnormalised
//                  accumulator) goes to the workspace.  head_dim 64 and 128.
//   decode_combine log-sum-exp merge of the chunks of each (layer, seq, head).
// K and V are read exactly once from HBM; softmax runs in base 2.
#include "sonic_dev.cuh"
#include "sonic_host.h"

namespace sonic {
namespace {

constexpr float kLn2 = 0.6931471805599453f;
constexpr float kLog2e = 1.4426950408889634f;

struct DecParams {
    const uint16_t *q;
    uint16_t *O;
    const int32_t *lens;
    const int32_t *kv_start;
    float *lse;
    float *part_acc;  // [units][max_chunks][D]
    float *part_ml;   // [units][max_chunks][2]
    // attention mass on Nexus keys (when nexus_mass is given): the role of
    // every key row, the output, and the per-chunk partial sums
    const uint8_t *role;
    float *nexus_mass;
    float *part_nx;   // [units][max_chunks]
    int32_t *status;
    int B, Hq, Hkv, G;
    int64_t total_kv_rows;  // rows of K_ret, V_ret (and role) per layer
    int64_t q_ls, o_ls;
    int chunk_len, max_chunks;
    float scale_log2;
};

// Maximum of v over the 32 lanes of the warp, in one instruction.
__device__ __forceinline__ float warp_max(float v) {
    float r;
    asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(v));
    return r;
}

// ---------------------------------------------------------------------------
// Tensor-core decode (head_dim 64 and 128).  Both contractions run on tcgen05 with the
// keys in the M dimension: S^T = K q^T (M = 128 keys of a tile, N = 16 query
// heads padded, K = D) and O^T += V^T P^T (M = D, N = 16, K = 128 keys, V read
// MN-major straight from the TMA stage).  Warp 0 streams K/V tiles through a
// 3-stage ring, warp 1 issues the MMAs, warps 2-5 (thread = key = TMEM lane)
// run a block-wide online softmax per head and write P (bf16) to shared
// memory; a running maximum that rises by less than 2^8 does not trigger an
// O rescale.  S^T and P are double buffered so S^T of the next tile overlaps
// the softmax and P.V of the current one.
//
// The kernel is persistent: one block per SM claims units (key chunk, KV
// head, sequence, layer) from a global counter (so ragged units balance over
// the SMs) and works through them as one continuous stream of key tiles: the
// K/V ring and the tensor pipe stay busy across unit boundaries (the next
// unit's q is staged and its first S^T issued while the current unit
// finishes).  q and the O^T accumulator are double buffered by unit.  Short
// sequences (a few tiles per unit) would otherwise spend most of a block's
// life on set-up and on the first copies.
// ---------------------------------------------------------------------------
constexpr int kTcKeys = 128;
constexpr int kTcStages = 3;
constexpr int kTcThreads = 192;
constexpr int kTcN = 16;  // query heads per MMA (padded)
constexpr float kTcRescale = 8.0f;

struct TcCfg {
    static constexpr int D = 128;
    static constexpr int kTileBytes = kTcKeys * D * 2;           // K or V tile: 32 KB
    static constexpr int kStageBytes = 2 * kTileBytes;           // 64 KB
    static constexpr int kQBufs = 2;                             // q of this unit and the next
    static constexpr int kOffQ = kTcStages * kStageBytes;        // q [2], 16 x 128 bf16, swizzled
    static constexpr int kQBytes = kTcN * D * 2;                 // 4 KB
    static constexpr int kOffP = kOffQ + kQBufs * kQBytes;       // P, [2][16 x 128 keys] bf16
    static constexpr int kPBytes = kTcN * kTcKeys * 2;           // 4 KB
    static constexpr int kOffRed = kOffP + 2 * kPBytes;          // [2][4][16] float
    static constexpr int kOffL = kOffRed + 2 * 4 * kTcN * 4;     // [4][16] float
    static constexpr int kOffN = kOffL + 4 * kTcN * 4;           // [4][16] float
    static constexpr int kOffBar = kOffN + 4 * kTcN * 4;
    static constexpr int kNumBars = 2 * kTcStages + 24;  // the pointers carved out below
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;
    static constexpr int kSeqCache = 1024;                       // sequences whose lens/kv_start
    static constexpr int kOffSeq = kOffMisc + 128;               // are cached: [2][1024] int32
    static constexpr size_t kSmem = 1024 + kOffSeq + 2 * kSeqCache * 4;
};
constexpr int kUnitSlots = 4;  // claimed-unit queue between the producer and the others

// Unit u: (key chunk, KV head, sequence, layer), KV head fastest.  A unit whose
// chunk starts past the sequence's end has no keys.
struct TcUnit {
    int u, kvh, chunk, b, layer, nkeys, ntiles, row0, len;
};

// The indices of unit w.u and its tile count (from w.nkeys).
__device__ __forceinline__ void tc_coords(const DecParams &p, int units_x, TcUnit &w) {
    const int x = w.u % units_x, y = w.u / units_x;
    w.kvh = x % p.Hkv;
    w.chunk = x / p.Hkv;
    w.b = y % p.B;
    w.layer = y / p.B;
    w.ntiles = (w.nkeys + kTcKeys - 1) / kTcKeys;
}

// seq_len / seq_start: the sequences' lengths and first rows cached in shared
// memory (B <= kSeqCache), or NULL to read them from global memory.
__device__ __forceinline__ bool tc_unit(const DecParams &p, int units_x, int u, TcUnit &w,
                                        const int32_t *seq_len, const int32_t *seq_start) {
    const int x = u % units_x, y = u / units_x;
    w.u = u;
    w.kvh = x % p.Hkv;
    w.chunk = x / p.Hkv;
    w.b = y % p.B;
    w.layer = y / p.B;
    int len = seq_len != nullptr ? seq_len[w.b] : p.lens[w.b];
    len = min(max(len, 0), p.max_chunks * p.chunk_len);
    const int start = seq_start != nullptr ? seq_start[w.b] : p.kv_start[w.b];
    if (start < 0 || (int64_t)start + len > p.total_kv_rows) {
        // rows outside the cache: the sequence is refused, nothing is read
        if (w.chunk == 0 && w.kvh == 0) set_status(p.status, SONIC_ERR_INVALID_ARGUMENT);
        len = 0;
    }
    const int key0 = w.chunk * p.chunk_len;
    w.len = len;
    w.nkeys = max(min(p.chunk_len, len - key0), 0);
    w.ntiles = (w.nkeys + kTcKeys - 1) / kTcKeys;
    w.row0 = start + key0;
    return w.nkeys > 0;
}

// D = 64 or 128.  The stage layout is the D = 128 one.  At D = 64 either the
// second 64-column half of each K and V tile is never loaded and stays zero
// (the ring is zeroed at kernel start), or (kPair, when G <= 8) a unit takes
// two KV heads: head 2i's rows fill the first half and head 2i+1's the second,
// the 16 staged query heads hold both heads' G queries, and S^T and O^T get a
// region per KV head (query column v belongs to head 2i for v < G, to head
// 2i+1 after), so a 128-key tile carries as many bytes as at D = 128 for the
// same per-tile softmax work.  O^T += V^T P^T keeps M = 128 either way (rows
// 64-127 accumulate zeros, or the other half's data; they are never written).
template <int D, int GT, bool kPair>
__global__ void __launch_bounds__(kTcThreads, 1)
decode_tc_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                 const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK16,
                 const __grid_constant__ CUtensorMap tmV16, const DecParams p, int units_x,
                 int n_units, int *unit_counter) {
    static_assert(D == 64 || D == 128, "head_dim 64 or 128");
    static_assert(!kPair || D == 64, "KV-head pairs at head_dim 64 only");
    constexpr int kHalves = D / 64;            // 64-column halves per K / V row
    constexpr int kLoads = kPair ? 2 : kHalves;  // 64-column boxes per K / V tile
    constexpr int kSStride = kPair ? 2 * kTcN : kTcN;  // TMEM columns of one S^T / O^T buffer
    constexpr uint32_t kTmemCols = kPair ? 128 : 64;
    using C = TcCfg;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t *q_s = smem + C::kOffQ;  // [2]
    uint8_t *P_s = smem + C::kOffP;  // [2]
    float *red = reinterpret_cast<float *>(smem + C::kOffRed);
    float *lred = reinterpret_cast<float *>(smem + C::kOffL);
    float *nred = reinterpret_cast<float *>(smem + C::kOffN);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + C::kOffBar);
    uint64_t *full = bars;                    // [stages] K/V tile landed
    uint64_t *empty = bars + kTcStages;       // [stages] its P.V is done
    uint64_t *s_full = bars + 2 * kTcStages;  // [2] per global tile
    uint64_t *p_full = s_full + 2;            // [2] per global tile: its P written (128 threads)
    uint64_t *o_done = p_full + 2;            // a P.V done
    uint64_t *mma_idle = o_done + 1;
    uint64_t *sm_sync = mma_idle + 1;  // the 128 softmax threads, once per tile
    uint64_t *ep_sync = sm_sync + 1;   // the 128 softmax threads, once per unit
    uint64_t *q_full = ep_sync + 1;    // [2] per unit: q staged
    uint64_t *q_empty = q_full + 2;    // [2] per unit: its last S^T done
    uint64_t *o_last = q_empty + 2;    // [2] per unit: its last P.V done
    uint64_t *o_free = o_last + 2;     // [2] per unit: its O^T read out (128 threads)
    uint64_t *uq_full = o_free + 2;    // [kUnitSlots] a claimed unit is in its slot
    uint64_t *uq_empty = uq_full + kUnitSlots;  // [kUnitSlots] the issuer and 4 warps read it
    int32_t *misc = reinterpret_cast<int32_t *>(smem + C::kOffMisc);
    // [kUnitSlots][4]: unit index (-1: no more), its keys, first key row, sequence length
    volatile int32_t *unit_q = misc + 4;
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + 1);

    const int G = p.G;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (timed_out(p.status)) return;
    if (tid == 0) {
        // a sequence longer than the plan allows is clipped, and reported
        for (int b = blockIdx.x; b < p.B; b += gridDim.x)
            if (p.lens[b] > p.max_chunks * p.chunk_len) set_status(p.status, SONIC_ERR_INVALID_ARGUMENT);
    }

    // The P buffers zeroed (rows >= GT stay zero), and the K/V ring: rows a
    // partial tile does not load keep older, finite data, which P = 0 cancels.
    for (int i = tid; i < 2 * C::kPBytes / 16; i += blockDim.x)
        reinterpret_cast<uint4 *>(P_s)[i] = make_uint4(0, 0, 0, 0);
    for (int i = tid; i < kTcStages * C::kStageBytes / 16; i += blockDim.x)
        reinterpret_cast<uint4 *>(smem)[i] = make_uint4(0, 0, 0, 0);
    // the sequences' lengths and first rows, for claiming units without
    // global loads on the producer's path
    int32_t *seq_len = nullptr, *seq_start = nullptr;
    if (p.B <= C::kSeqCache) {
        seq_len = reinterpret_cast<int32_t *>(smem + C::kOffSeq);
        seq_start = seq_len + C::kSeqCache;
        for (int b = tid; b < p.B; b += blockDim.x) {
            seq_len[b] = p.lens[b];
            seq_start[b] = p.kv_start[b];
        }
    }
    if (tid == 0) {
        for (int s = 0; s < kTcStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&s_full[i], 1);
            mbar_init(&p_full[i], 128);
            mbar_init(&o_last[i], 1);
            mbar_init(&o_free[i], 128);
        }
        for (int i = 0; i < C::kQBufs; ++i) {
            mbar_init(&q_full[i], 1);
            mbar_init(&q_empty[i], 1);
        }
        for (int i = 0; i < kUnitSlots; ++i) {
            mbar_init(&uq_full[i], 1);
            mbar_init(&uq_empty[i], 5);
        }
        mbar_init(o_done, 1);
        mbar_init(mma_idle, 1);
        mbar_init(sm_sync, 128);
        mbar_init(ep_sync, 128);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(reinterpret_cast<uint32_t *>(&misc[0]), kTmemCols);
        tmem_relinquish();
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = static_cast<uint32_t>(misc[0]);
    // TMEM: S^T [2] then O^T [2], kSStride columns each (a 16-column region
    // per KV head of the unit)
    const uint32_t tS = tmem, tO = tmem + 2 * kSStride;
    const int Gv = kPair ? 2 * G : G;  // query columns of a unit
    // The k-th claimed unit (w.u = -1: none left, or a wait gave up), from
    // shared memory: the consumers never touch global memory for it.  Each
    // reader (the issuer, lane 0 of each softmax warp) frees the slot.
    auto read_unit = [&](int k, TcUnit &w) -> bool {
        const int slot = k & (kUnitSlots - 1);
        w.u = -1;
        if (!mbar_wait(&uq_full[slot], (k / kUnitSlots) & 1, p.status, abort_flag)) return false;
        const volatile int32_t *q = unit_q + slot * 4;
        w.u = q[0];
        w.nkeys = q[1];
        w.row0 = q[2];
        w.len = q[3];
        mbar_arrive(&uq_empty[slot]);
        return w.u >= 0;
    };

    int issued_q = 0, issued_kv = 0;  // copies the producer issued (for the drain)
    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&tmK);
            tma_prefetch_desc(&tmV);
        }
        // Lane 0 claims units from the counter, publishes each in the unit
        // queue and streams its q (one TMA box of 16 heads: rows past the
        // group's G heads are other heads' q or zeros, whose S^T columns the
        // softmax never reads) and its K/V tiles.  The claim of unit k + 1 is
        // sent before unit k's copies are queued; its answer is needed only
        // after them.
        if (lane == 0) {
            tma_prefetch_desc(&tmQ);
            int T = 0;  // K/V tiles issued
            int pending = atomicAdd(unit_counter, 1);
            for (int k = 0;; ++k) {
                const int slot = k & (kUnitSlots - 1);
                bool ok = k < kUnitSlots ||
                          mbar_wait(&uq_empty[slot], ((k / kUnitSlots) - 1) & 1, p.status, abort_flag);
                int u = -1;
                TcUnit w;
                if (ok) {
                    u = pending;
                    while (u < n_units && !tc_unit(p, units_x, u, w, seq_len, seq_start))
                        u = atomicAdd(unit_counter, 1);
                    if (u >= n_units) u = -1;
                }
                volatile int32_t *q = unit_q + slot * 4;
                q[0] = u;
                q[1] = w.nkeys;
                q[2] = w.row0;
                q[3] = w.len;
                mbar_arrive(&uq_full[slot]);  // release: the slot is written
                if (u < 0) break;
                pending = atomicAdd(unit_counter, 1);
                // q into buffer k & 1 once the S^T MMAs of unit k - 2 no longer read it
                const int qb = k & 1;
                if (k >= 2 && !mbar_wait(&q_empty[qb], ((k >> 1) - 1) & 1, p.status, abort_flag))
                    break;
                const int kvh0 = kPair ? 2 * w.kvh : w.kvh;  // first KV head of the unit
                mbar_arrive_expect_tx(&q_full[qb], kHalves * (kTcN * 128));
#pragma unroll
                for (int hh = 0; hh < kHalves; ++hh)
                    tma_load_4d(q_s + qb * C::kQBytes + hh * (kTcN * 128), &tmQ, &q_full[qb],
                                hh * 64, kvh0 * G, w.b, w.layer);
                issued_q = k + 1;
                for (int t = 0; t < w.ntiles; ++t, ++T) {
                    const int s = T % kTcStages;
                    if (T >= kTcStages &&
                        !mbar_wait(&empty[s], ((T / kTcStages) - 1) & 1, p.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    uint8_t *kd = smem + s * C::kStageBytes;
                    uint8_t *vd = kd + C::kTileBytes;
                    const int r = w.row0 + t * kTcKeys;
                    const int rem = w.nkeys - t * kTcKeys;
                    if (rem >= kTcKeys) {
                        mbar_arrive_expect_tx(&full[s], 2 * kLoads * (kTcKeys * 128));
#pragma unroll
                        for (int hh = 0; hh < kLoads; ++hh) {
                            const int dc = kPair ? 0 : hh * 64, hc = kPair ? kvh0 + hh : kvh0;
                            tma_load_4d(kd + hh * (kTcKeys * 128), &tmK, &full[s], dc, hc, r,
                                        w.layer);
                            tma_load_4d(vd + hh * (kTcKeys * 128), &tmV, &full[s], dc, hc, r,
                                        w.layer);
                        }
                    } else {
                        // a unit's last, partial tile: only its rows, in 16-row boxes
                        // (the rows past them keep older data; the softmax masks
                        // their scores and zeroes their V rows)
                        const int nb = (rem + 15) / 16;
                        mbar_arrive_expect_tx(&full[s], nb * 2 * kLoads * (16 * 128));
                        for (int j = 0; j < nb; ++j)
#pragma unroll
                            for (int hh = 0; hh < kLoads; ++hh) {
                                const int dc = kPair ? 0 : hh * 64, hc = kPair ? kvh0 + hh : kvh0;
                                tma_load_4d(kd + hh * (kTcKeys * 128) + j * (16 * 128), &tmK16,
                                            &full[s], dc, hc, r + 16 * j, w.layer);
                                tma_load_4d(vd + hh * (kTcKeys * 128) + j * (16 * 128), &tmV16,
                                            &full[s], dc, hc, r + 16 * j, w.layer);
                            }
                    }
                }
                if (!ok) break;
            }
            issued_kv = T;
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idS = idesc_bf16_f32(kTcKeys, kTcN, 0, 0);
            constexpr uint32_t idPV = idesc_bf16_f32(128, kTcN, 0, 1);  // M = 128 at D = 64 too
            const uint32_t base = smem_u32(smem), q_base = smem_u32(q_s), p_addr = smem_u32(P_s);
            // S^T of global tile T (unit number k, its tile t) from q buffer k % 2
            auto issue_s = [&](int T, int k, int t, int nt) -> bool {
                if (t == 0 &&
                    !mbar_wait(&q_full[k % C::kQBufs], (k / C::kQBufs) & 1, p.status, abort_flag))
                    return false;
                if (!mbar_wait(&full[T % kTcStages], (T / kTcStages) & 1, p.status, abort_flag))
                    return false;
                tc_fence_after();
                const uint32_t k_addr = base + (T % kTcStages) * C::kStageBytes;
                const uint32_t q_addr = q_base + (k % C::kQBufs) * C::kQBytes;
                const uint32_t sbuf = tS + (T & 1) * kSStride;
                if (kPair) {
                    // one S^T region per KV head: its K half against all staged queries
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh)
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            tc_mma_ss(sbuf + hh * kTcN,
                                      smem_desc_sw128(k_addr + hh * (kTcKeys * 128) + kk * 32, 16,
                                                      1024),
                                      smem_desc_sw128(q_addr + kk * 32, 16, 1024), idS,
                                      kk > 0 ? 1u : 0u);
                } else {
#pragma unroll
                    for (int kk = 0; kk < D / 16; ++kk) {
                        const uint64_t a = smem_desc_sw128(
                            k_addr + (kk >> 2) * (kTcKeys * 128) + (kk & 3) * 32, 16, 1024);
                        const uint64_t bd = smem_desc_sw128(
                            q_addr + (kk >> 2) * (kTcN * 128) + (kk & 3) * 32, 16, 1024);
                        tc_mma_ss(sbuf, a, bd, idS, kk > 0 ? 1u : 0u);
                    }
                }
                tc_commit(&s_full[T & 1]);
                if (t == nt - 1) tc_commit(&q_empty[k % C::kQBufs]);
                return true;
            };
            TcUnit w, nx;
            int T = 0, k = 0;
            bool ok = read_unit(0, w);
            if (ok) {
                tc_coords(p, units_x, w);
                ok = issue_s(0, 0, 0, w.ntiles);
            }
            for (bool more = true; ok && more; ++k) {
                bool has_next = false;
                for (int t = 0; ok && t < w.ntiles; ++t, ++T) {
                    // The next tile: this unit's, or the next unit's first (read
                    // only now: the producer publishes it after queueing all of this
                    // unit's copies).  Its S^T goes before this tile's P.V when its
                    // K tile (and q) are already in; otherwise after, so that a late
                    // copy never holds back the P.V that frees a stage.
                    int nk = k, nt1 = t + 1, nnt = w.ntiles;
                    bool next_tile = t + 1 < w.ntiles;
                    if (!next_tile) {
                        has_next = read_unit(k + 1, nx);
                        if (has_next) {
                            tc_coords(p, units_x, nx);
                            next_tile = true;
                            nk = k + 1;
                            nt1 = 0;
                            nnt = nx.ntiles;
                        }
                    }
                    bool s_issued = false;
                    if (next_tile &&
                        mbar_test(&full[(T + 1) % kTcStages], ((T + 1) / kTcStages) & 1) &&
                        (nt1 > 0 || mbar_test(&q_full[nk & 1], (nk >> 1) & 1))) {
                        ok = issue_s(T + 1, nk, nt1, nnt);
                        s_issued = true;
                    }
                    if (!ok || !mbar_wait(&p_full[T & 1], (T >> 1) & 1, p.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    // O^T buffer k & 1: unit k - 2's epilogue has read it out
                    if (t == 0 && k >= 2 &&
                        !mbar_wait(&o_free[k & 1], ((k >> 1) - 1) & 1, p.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t v_addr = base + (T % kTcStages) * C::kStageBytes + C::kTileBytes;
                    const uint32_t pb = p_addr + (T & 1) * C::kPBytes;
#pragma unroll
                    for (int hh = 0; hh < (kPair ? 2 : 1); ++hh)
#pragma unroll
                        for (int kk = 0; kk < kTcKeys / 16; ++kk) {
                            const uint64_t a = smem_desc_sw128(
                                v_addr + hh * (kTcKeys * 128) + kk * (16 * 128), kTcKeys * 128, 1024);
                            const uint64_t bd = smem_desc_sw128(
                                pb + (kk >> 2) * (kTcN * 128) + (kk & 3) * 32, 16, 1024);
                            tc_mma_ss(tO + (k & 1) * kSStride + hh * kTcN, a, bd, idPV,
                                      (t > 0 || kk > 0) ? 1u : 0u);
                        }
                    tc_commit(o_done);
                    tc_commit(&empty[T % kTcStages]);
                    if (t == w.ntiles - 1) tc_commit(&o_last[k & 1]);
                    if (next_tile && !s_issued) ok = issue_s(T + 1, nk, nt1, nnt);
                }
                more = has_next;
                w = nx;
            }
            // every MMA issued by this thread has finished once this arrives (a
            // wait bounded by time alone: tensor memory is freed after it)
            tc_commit(mma_idle);
            mbar_drain(mma_idle, 0);
        }
    } else {
        // ------------------------------------------------------------ softmax
        const int quarter = warp & 3;
        const int r = quarter * 32 + lane;  // key row of the tile, and d row of O^T
        const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
        // Unit epilogue: normalise O^T of unit k and write it (or its partial).
        // It runs one tile into the next unit, when the unit's last P.V is long
        // done, so the move from one unit to the next costs no pipeline drain.
        const bool want_nx = p.nexus_mass != nullptr;
        auto epilogue = [&](const TcUnit &w, int k, const float (&m)[GT], const float (&l)[GT],
                            const float (&n)[GT]) -> bool {
            const uint32_t tOk = tO + (k & 1) * kSStride;
            if (!mbar_wait(&o_last[k & 1], (k >> 1) & 1, p.status, abort_flag)) return false;
            tc_fence_after();
#pragma unroll
            for (int g = 0; g < GT; ++g) {
                float v = l[g], vn = n[g];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    v += __shfl_xor_sync(0xffffffffu, v, o);
                    if (want_nx) vn += __shfl_xor_sync(0xffffffffu, vn, o);
                }
                if (lane == 0) {
                    lred[quarter * kTcN + g] = v;
                    nred[quarter * kTcN + g] = vn;
                }
            }
            mbar_arrive(ep_sync);
            if (!mbar_wait(ep_sync, k & 1, p.status, abort_flag)) return false;
            uint32_t o[16];
            tmem_ld16(tOk + lane_base, o);
            if (kPair) {  // query columns v >= G: the second KV head's region
                uint32_t ob[16];
                tmem_ld16(tOk + lane_base + kTcN, ob);
                tmem_ld_wait();
                reg_fence16(ob);
#pragma unroll
                for (int g = 0; g < 16; ++g)
                    if (g >= G) o[g] = ob[g];
            }
            tmem_ld_wait();
            reg_fence16(o);
            float Lg[GT], Ng[GT];
#pragma unroll
            for (int g = 0; g < GT; ++g) {
                Lg[g] = lred[g] + lred[kTcN + g] + lred[2 * kTcN + g] + lred[3 * kTcN + g];
                Ng[g] = nred[g] + nred[kTcN + g] + nred[2 * kTcN + g] + nred[3 * kTcN + g];
            }
            // O^T of this unit is in registers and lred read: the buffers are free
            tc_fence_before();
            mbar_arrive(&o_free[k & 1]);
            const int n_chunks = (w.len + p.chunk_len - 1) / p.chunk_len;
            const int hb = (kPair ? 2 * w.kvh : w.kvh) * G;  // the unit's first query head
            const int64_t unit0 = ((int64_t)w.layer * p.B + w.b) * p.Hq + hb;
#pragma unroll
            for (int g = 0; g < GT; ++g) {
                if (g >= Gv) break;
                const float L = Lg[g];
                const float a = __uint_as_float(o[g]);
                if (n_chunks == 1) {
                    uint16_t *op =
                        p.O + w.layer * p.o_ls + ((int64_t)w.b * p.Hq + hb + g) * D;
                    if (r < D) op[r] = __bfloat16_as_ushort(__float2bfloat16_rn(a / L));
                    if (r == 0 && p.lse != nullptr) p.lse[unit0 + g] = (m[g] + __log2f(L)) * kLn2;
                    if (r == 0 && want_nx) p.nexus_mass[unit0 + g] = Ng[g] / L;
                } else {
                    const int64_t slot = (unit0 + g) * p.max_chunks + w.chunk;
                    if (r < D) p.part_acc[slot * D + r] = a;
                    if (r == 0) {
                        p.part_ml[slot * 2 + 0] = m[g];
                        p.part_ml[slot * 2 + 1] = L;
                        if (want_nx) p.part_nx[slot] = Ng[g];
                    }
                }
            }
            return true;
        };
        bool ok = true, pend = false;  // pend: unit kp still owes its epilogue
        int T = 0, kp = 0;
        TcUnit wp;
        float mp[GT], lp[GT], np[GT];
        for (int k = 0; ok; ++k) {
            TcUnit w;
            if (lane == 0) read_unit(k, w);
            w.u = __shfl_sync(0xffffffffu, w.u, 0);
            if (w.u < 0) break;
            w.nkeys = __shfl_sync(0xffffffffu, w.nkeys, 0);
            w.row0 = __shfl_sync(0xffffffffu, w.row0, 0);
            w.len = __shfl_sync(0xffffffffu, w.len, 0);
            tc_coords(p, units_x, w);
            const uint32_t tOk = tO + (k & 1) * kSStride;
            float m[GT], l[GT], n[GT];
#pragma unroll
            for (int g = 0; g < GT; ++g) {
                m[g] = -INFINITY;
                l[g] = 0.f;
                n[g] = 0.f;
            }
            for (int t = 0; t < w.ntiles; ++t, ++T) {
                // this key's role, loaded before the wait (kept rows only)
                const bool in_unit = t * kTcKeys + r < w.nkeys;
                int role_k = 255;
                if (want_nx && in_unit) role_k = p.role[w.row0 + t * kTcKeys + r];
                if (!mbar_wait(&s_full[T & 1], (T >> 1) & 1, p.status, abort_flag)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                uint32_t sr[16];
                tmem_ld16(tS + lane_base + (T & 1) * kSStride, sr);
                if (kPair) {  // query columns v >= G: the second KV head's region
                    uint32_t sb[16];
                    tmem_ld16(tS + lane_base + (T & 1) * kSStride + kTcN, sb);
                    tmem_ld_wait();
                    reg_fence16(sb);
#pragma unroll
                    for (int g = 0; g < 16; ++g)
                        if (g >= G) sr[g] = sb[g];
                }
                tmem_ld_wait();
                reg_fence16(sr);
                const bool valid = in_unit;
                const bool isn = role_k == SONIC_ROLE_NEXUS;
                float sv[GT];
                float *rd = red + (T & 1) * 4 * kTcN;
#pragma unroll
                for (int g = 0; g < GT; ++g) {
                    sv[g] = valid ? __uint_as_float(sr[g]) * p.scale_log2 : -INFINITY;
                    const float wm = warp_max(sv[g]);
                    if (lane == 0) rd[quarter * kTcN + g] = wm;
                }
                // all four warps' maxima visible (bounded: a wait that gives up ends the loop)
                mbar_arrive(sm_sync);
                if (!mbar_wait(sm_sync, T & 1, p.status, abort_flag)) {
                    ok = false;
                    break;
                }
                float alpha[GT];
                bool resc = false;
#pragma unroll
                for (int g = 0; g < GT; ++g) {
                    const float mt = fmaxf(fmaxf(rd[g], rd[kTcN + g]),
                                           fmaxf(rd[2 * kTcN + g], rd[3 * kTcN + g]));
                    alpha[g] = 1.f;
                    if (t == 0) {
                        m[g] = mt;
                    } else if (mt > m[g] + kTcRescale) {
                        alpha[g] = ex2(m[g] - mt);
                        m[g] = mt;
                        resc = true;
                    }
                }
                // P^T column r (this key) in the swizzled K-major P buffer
                uint8_t *pb = P_s + (T & 1) * C::kPBytes + (r >> 6) * (kTcN * 128) + (r & 7) * 2;
                const int jj = (r & 63) >> 3;
#pragma unroll
                for (int g = 0; g < GT; ++g) {
                    // the row sum adds the rounded probability P.V multiplies by
                    const __nv_bfloat16 pr = __float2bfloat16_rn(ex2(sv[g] - m[g]));
                    l[g] = l[g] * alpha[g] + __bfloat162float(pr);
                    if (want_nx) n[g] = n[g] * alpha[g] + (isn ? __bfloat162float(pr) : 0.f);
                    *reinterpret_cast<__nv_bfloat16 *>(pb + g * 128 + ((jj ^ (g & 7)) << 4)) = pr;
                }
                if (!valid && r < ((w.nkeys - t * kTcKeys + 15) & ~15)) {
                    // rows a partial tile loaded past the unit's keys (another
                    // sequence's, or junk): zero their V, so 0 * garbage cannot
                    // reach O
                    uint8_t *vrow =
                        smem + (T % kTcStages) * C::kStageBytes + C::kTileBytes + r * 128;
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh)
#pragma unroll
                        for (int u = 0; u < 8; ++u)
                            reinterpret_cast<uint4 *>(vrow + hh * (kTcKeys * 128))[u] =
                                make_uint4(0, 0, 0, 0);
                }
                if (resc) {  // block-uniform
                    if (!mbar_wait(o_done, (T - 1) & 1, p.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
#pragma unroll
                    for (int hh = 0; hh < (kPair ? 2 : 1); ++hh) {
                        uint32_t o[16];
                        tmem_ld16(tOk + lane_base + hh * kTcN, o);
                        tmem_ld_wait();
                        reg_fence16(o);
#pragma unroll
                        for (int g = 0; g < GT; ++g)
                            o[g] = __float_as_uint(__uint_as_float(o[g]) * alpha[g]);
                        tmem_st16(tOk + lane_base + hh * kTcN, o);
                    }
                    tmem_st_wait();
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(&p_full[T & 1]);
                if (t == 0 && pend) {
                    ok = epilogue(wp, kp, mp, lp, np);
                    pend = false;
                    if (!ok) break;
                }
            }
            if (!ok) break;
            wp = w;
            kp = k;
#pragma unroll
            for (int g = 0; g < GT; ++g) {
                mp[g] = m[g];
                lp[g] = l[g];
                np[g] = n[g];
            }
            pend = true;
        }
        if (ok && pend) epilogue(wp, kp, mp, lp, np);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // After an abort no thread waits any more; let the copies the producer
    // issued land before the block's shared memory goes away (older ones have:
    // their buffers were waited free before being refilled).
    if (*abort_flag && warp == 0 && lane == 0) {
        for (int k = max(0, issued_q - C::kQBufs); k < issued_q; ++k)
            mbar_drain(&q_full[k % C::kQBufs], (k / C::kQBufs) & 1);
        for (int u = max(0, issued_kv - kTcStages); u < issued_kv; ++u)
            mbar_drain(&full[u % kTcStages], (u / kTcStages) & 1);
    }
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// One warp per (layer, sequence, query head).
template <int D>
__global__ void __launch_bounds__(128)
decode_combine_kernel(const DecParams p, int n_layers) {
    const int64_t unit = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t n_units = (int64_t)n_layers * p.B * p.Hq;
    if (unit >= n_units) return;
    const int h = (int)(unit % p.Hq);
    const int64_t lb = unit / p.Hq;
    const int b = (int)(lb % p.B), layer = (int)(lb / p.B);
    const int len = min(p.lens[b], p.max_chunks * p.chunk_len);
    const int n_chunks = (len + p.chunk_len - 1) / p.chunk_len;
    if (n_chunks == 1) return;  // written by the split kernel
    uint16_t *op = p.O + layer * p.o_ls + ((int64_t)b * p.Hq + h) * D;
    constexpr int kDpl = D / 32;
    if (n_chunks <= 0) {
#pragma unroll
        for (int e = 0; e < kDpl; ++e) op[lane * kDpl + e] = 0;
        if (lane == 0 && p.lse != nullptr) p.lse[unit] = -INFINITY;
        if (lane == 0 && p.nexus_mass != nullptr) p.nexus_mass[unit] = 0.f;
        return;
    }
    const float *ml = p.part_ml + unit * p.max_chunks * 2;
    const float *ac = p.part_acc + unit * p.max_chunks * D;
    float M = -INFINITY;
    for (int c = lane; c < n_chunks; c += 32) M = fmaxf(M, ml[2 * c]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    float L = 0.f, N = 0.f;
    float a[kDpl];
#pragma unroll
    for (int e = 0; e < kDpl; ++e) a[e] = 0.f;
    for (int c = 0; c < n_chunks; ++c) {
        const float f = ex2(ml[2 * c] - M);
        L += f * ml[2 * c + 1];
        if (p.nexus_mass != nullptr) N += f * p.part_nx[unit * p.max_chunks + c];
#pragma unroll
        for (int e = 0; e < kDpl; ++e) a[e] += f * ac[(int64_t)c * D + lane * kDpl + e];
    }
#pragma unroll
    for (int e = 0; e < kDpl; ++e)
        op[lane * kDpl + e] = __bfloat16_as_ushort(__float2bfloat16_rn(a[e] / L));
    if (lane == 0 && p.lse != nullptr) p.lse[unit] = (M + __log2f(L)) * kLn2;
    if (lane == 0 && p.nexus_mass != nullptr) p.nexus_mass[unit] = N / L;
}

// Every output of a call with no key rows at all: O = 0, lse = -inf, mass 0.
__global__ void decode_empty_kernel(uint16_t *O, int64_t o_ls, float *lse, float *nexus_mass,
                                    int n_layers, int64_t per_layer_units, int D) {
    const int64_t n = (int64_t)n_layers * per_layer_units;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n * D;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t unit = i / D, layer = unit / per_layer_units;
        O[layer * o_ls + (unit - layer * per_layer_units) * D + (i - unit * D)] = 0;
        if (i - unit * D == 0) {
            if (lse != nullptr) lse[unit] = -INFINITY;
            if (nexus_mass != nullptr) nexus_mass[unit] = 0.f;
        }
    }
}

int g_template(int G) {
    if (G <= 1) return 1;
    if (G <= 2) return 2;
    if (G <= 4) return 4;
    if (G <= 7) return 7;
    if (G <= 8) return 8;
    if (G <= 16) return 16;
    return 0;
}

struct Plan {
    int chunk_len, max_chunks;
    // partial accumulators, partial (max, sum), partial Nexus sums, unit counter
    size_t ws_acc, ws_ml, ws_nx, ws_cnt;
    size_t total() const { return ws_acc + ws_ml + ws_nx + ws_cnt; }
};

// head_dim 64 with G <= 8 and an even number of KV heads: units of two KV heads.
bool use_pairs(const sonic_decode_args *a) {
    if (a->n_heads_kv <= 0 || a->n_heads_q % a->n_heads_kv != 0) return false;
    const int G = a->n_heads_q / a->n_heads_kv;
    return a->head_dim == 64 && G <= 8 && a->n_heads_kv % 2 == 0;
}

Plan make_plan(const sonic_decode_args *a) {
    Plan pl{};
    const int kv_units = a->n_heads_kv / (use_pairs(a) ? 2 : 1);  // KV heads (or pairs) per unit row
    const int max_len = a->max_len > 0 ? a->max_len : 1;
    // explicit split lengths are rounded up to the kernel's key tile
    const int tile = kTcKeys;
    const long long c0 = a->chunk_len < max_len ? a->chunk_len : max_len;
    int C = (int)((c0 + tile - 1) / tile * tile);
    if (C <= 0) {
        const long long units = (long long)a->batch * kv_units * a->n_layers;
        const long long target = 4LL * device_sm_count();
        long long splits = units >= target ? 1 : (target + units - 1) / units;
        long long c = (max_len + splits - 1) / splits;
        c = (c + 255) / 256 * 256;
        C = (int)(c < 256 ? 256 : c);
    }
    pl.chunk_len = C;
    pl.max_chunks = (max_len + C - 1) / C;
    const size_t units_q = (size_t)a->batch * a->n_heads_q * a->n_layers;
    if (pl.max_chunks > 1) {
        pl.ws_acc = round_up(units_q * pl.max_chunks * a->head_dim * sizeof(float), 256);
        pl.ws_ml = round_up(units_q * pl.max_chunks * 2 * sizeof(float), 256);
        if (a->nexus_mass != nullptr)
            pl.ws_nx = round_up(units_q * pl.max_chunks * sizeof(float), 256);
    }
    pl.ws_cnt = 256;  // the persistent kernel's unit counter
    return pl;
}

// Persistent launch: one block per SM (the stage ring takes most of shared
// memory); the blocks claim units from a counter zeroed on the stream first.
struct TcMaps {
    CUtensorMap k, v, q, k16, v16;
};

template <int D, int GT, bool kPair>
cudaError_t launch_tc(const TcMaps &m, const DecParams &p, int units_x, int n_units, int *counter,
                      cudaStream_t stream) {
    constexpr size_t smem = TcCfg::kSmem;
    static_assert(smem <= 232448, "decode shared memory");
    auto kern = decode_tc_kernel<D, GT, kPair>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(counter, 0, sizeof(int), stream);
    if (e != cudaSuccess) return e;
    const int sms = device_sm_count();
    const int blocks = n_units < sms ? n_units : sms;
    kern<<<blocks, kTcThreads, smem, stream>>>(m.k, m.v, m.q, m.k16, m.v16, p, units_x, n_units,
                                               counter);
    return cudaGetLastError();
}

template <int D, bool kPair>
cudaError_t dispatch_tc(int GT, const TcMaps &m, const DecParams &p, int units_x, int n_units,
                        int *counter, cudaStream_t s) {
    switch (GT) {
        case 1: return launch_tc<D, 1, kPair>(m, p, units_x, n_units, counter, s);
        case 2: return launch_tc<D, 2, kPair>(m, p, units_x, n_units, counter, s);
        case 4: return launch_tc<D, 4, kPair>(m, p, units_x, n_units, counter, s);
        case 7: return launch_tc<D, 7, kPair>(m, p, units_x, n_units, counter, s);
        case 8: return launch_tc<D, 8, kPair>(m, p, units_x, n_units, counter, s);
        case 16: return launch_tc<D, 16, kPair>(m, p, units_x, n_units, counter, s);
    }
    return cudaErrorInvalidValue;
}



}  // namespace
}  // namespace sonic

using namespace sonic;

extern "C" size_t sonic_decode_workspace_size(const sonic_decode_args *a) {
    if (a == nullptr || a->batch <= 0 || a->n_layers < 1 || a->n_heads_q < 1 ||
        a->head_dim < 1)
        return 0;
    Plan pl = make_plan(a);
    return pl.total();
}

extern "C" sonic_status_t sonic_attn_decode(const uint16_t *q, const uint16_t *K_ret,
                                            const uint16_t *V_ret, const int32_t *lens,
                                            uint16_t *O, const sonic_decode_args *a,
                                            sonic_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (a == nullptr) return SONIC_ERR_INVALID_ARGUMENT;
    if (a->batch < 0 || a->n_layers < 1 || a->n_heads_kv < 1 || a->n_heads_q < 1 ||
        a->n_heads_q % a->n_heads_kv != 0 || a->max_len < 0 || a->total_kv_rows < 0)
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->batch == 0) return SONIC_OK;
    if (q == nullptr || K_ret == nullptr || V_ret == nullptr || lens == nullptr ||
        O == nullptr || a->kv_start == nullptr)
        return SONIC_ERR_INVALID_ARGUMENT;
    const int D = a->head_dim;
    if (D != 64 && D != 128) return SONIC_ERR_UNSUPPORTED;
    const int G = a->n_heads_q / a->n_heads_kv;
    const int GT = g_template(G);
    if (GT == 0) return SONIC_ERR_UNSUPPORTED;
    if (a->chunk_len < 0) return SONIC_ERR_INVALID_ARGUMENT;
    if (a->nexus_mass != nullptr && a->role == nullptr) return SONIC_ERR_INVALID_ARGUMENT;
    if (!aligned16(K_ret) || !aligned16(V_ret) || !aligned16(q) || (a->q_layer_stride * 2) % 16)
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->n_layers > 1 && (a->kv_layer_stride <= 0 || (a->kv_layer_stride * 2) % 16 != 0))
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->total_kv_rows == 0 || a->max_len == 0) {
        // nothing to attend: every output is zero (lse -inf)
        const long long units = (long long)a->batch * a->n_heads_q;
        const long long n = units * a->n_layers * D;
        const unsigned blocks = (unsigned)(n / 256 + 1 < 4096 ? n / 256 + 1 : 4096);
        decode_empty_kernel<<<blocks, 256, 0, stream>>>(O, a->o_layer_stride, a->lse,
                                                       a->nexus_mass, a->n_layers, units, D);
        return cudaGetLastError() == cudaSuccess ? SONIC_OK : SONIC_ERR_CUDA;
    }
    Plan pl = make_plan(a);
    const size_t need = pl.total();
    if (need > 0 && (a->workspace == nullptr || a->workspace_bytes < need))
        return SONIC_ERR_WORKSPACE;
    const bool pairs = use_pairs(a);
    const long long units_x = (long long)pl.max_chunks * (a->n_heads_kv / (pairs ? 2 : 1));
    if (units_x > 0x7fffffffLL ||
        units_x * a->batch * a->n_layers > 0x7fffffffLL)
        return SONIC_ERR_UNSUPPORTED;

    const uint64_t row_elems = (uint64_t)a->n_heads_kv * D;
    const uint64_t layer_bytes = a->n_layers > 1 ? (uint64_t)a->kv_layer_stride * 2
                                                 : (uint64_t)a->total_kv_rows * row_elems * 2;
    const uint64_t dims[4] = {(uint64_t)D, (uint64_t)a->n_heads_kv, (uint64_t)a->total_kv_rows,
                              (uint64_t)a->n_layers};
    const uint64_t strides[3] = {(uint64_t)D * 2, row_elems * 2, layer_bytes};
    const uint32_t box[4] = {64, 1, (uint32_t)kTcKeys, 1};
    CUtensorMap tk, tv;
    TcMaps tm{};
    if (!make_tmap_bf16_4d(&tk, K_ret, dims, strides, box) ||
        !make_tmap_bf16_4d(&tv, V_ret, dims, strides, box))
        return SONIC_ERR_INVALID_ARGUMENT;
    {
        tm.k = tk;
        tm.v = tv;
        const uint32_t box16[4] = {64, 1, 16, 1};
        if (!make_tmap_bf16_4d(&tm.k16, K_ret, dims, strides, box16) ||
            !make_tmap_bf16_4d(&tm.v16, V_ret, dims, strides, box16))
            return SONIC_ERR_INVALID_ARGUMENT;
        // q as (D, head, sequence, layer): one box = 16 heads of one sequence
        const uint64_t qdims[4] = {(uint64_t)D, (uint64_t)a->n_heads_q, (uint64_t)a->batch,
                                   (uint64_t)a->n_layers};
        const uint64_t qstr[3] = {(uint64_t)D * 2, (uint64_t)a->n_heads_q * D * 2,
                                  a->n_layers > 1 ? (uint64_t)a->q_layer_stride * 2
                                                  : (uint64_t)a->batch * a->n_heads_q * D * 2};
        const uint32_t qbox[4] = {64, (uint32_t)kTcN, 1, 1};
        if (!make_tmap_bf16_4d(&tm.q, q, qdims, qstr, qbox)) return SONIC_ERR_INVALID_ARGUMENT;
    }

    DecParams p{};
    p.q = q;
    p.O = O;
    p.lens = lens;
    p.kv_start = a->kv_start;
    p.lse = a->lse;
    p.part_acc = static_cast<float *>(a->workspace);
    p.part_ml = reinterpret_cast<float *>(static_cast<char *>(a->workspace) + pl.ws_acc);
    p.part_nx =
        reinterpret_cast<float *>(static_cast<char *>(a->workspace) + pl.ws_acc + pl.ws_ml);
    p.role = a->role;
    p.nexus_mass = a->nexus_mass;
    p.status = a->status;
    p.B = a->batch;
    p.Hq = a->n_heads_q;
    p.Hkv = a->n_heads_kv / (pairs ? 2 : 1);  // units per (chunk, sequence, layer)
    p.total_kv_rows = a->total_kv_rows;
    p.G = G;
    p.q_ls = a->q_layer_stride;
    p.o_ls = a->o_layer_stride;
    p.chunk_len = pl.chunk_len;
    p.max_chunks = pl.max_chunks;
    const float scale = a->softmax_scale > 0.f ? a->softmax_scale : 1.0f / sqrtf((float)D);
    p.scale_log2 = scale * kLog2e;

    int *counter = reinterpret_cast<int *>(static_cast<char *>(a->workspace) + pl.ws_acc +
                                           pl.ws_ml + pl.ws_nx);
    const int n_units = (int)(units_x * a->batch * a->n_layers);
    cudaError_t e =
        D == 128 ? dispatch_tc<128, false>(GT, tm, p, (int)units_x, n_units, counter, stream)
        : pairs  ? dispatch_tc<64, true>(g_template(2 * G), tm, p, (int)units_x, n_units, counter,
                                         stream)
                 : dispatch_tc<64, false>(GT, tm, p, (int)units_x, n_units, counter, stream);
    if (e != cudaSuccess) return SONIC_ERR_CUDA;
    const long long units = (long long)a->n_layers * a->batch * a->n_heads_q;
    const unsigned cblocks = (unsigned)((units * 32 + 127) / 128);
    if (D == 128)
        decode_combine_kernel<128><<<cblocks, 128, 0, stream>>>(p, a->n_layers);
    else
        decode_combine_kernel<64><<<cblocks, 128, 0, stream>>>(p, a->n_layers);
    return cudaGetLastError() == cudaSuccess ? SONIC_OK : SONIC_ERR_CUDA;
}
