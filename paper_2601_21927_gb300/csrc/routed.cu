// Role-routed linear map: Y = X W^T on ordinary rows and X W_N^T on Nexus
// rows (Sec. 3.1: Nexus tokens have dedicated projection matrices W_Q^N,
// W_K^N, W_V^N, W_O^N), with the output columns cut into parts that go to
// buffers of their own, each at the row itself or at a caller-given row (so
// the K and V of new tokens land straight in their retained-cache rows).
//
// Launches, none of which needs a host round trip:
//   role_count    per 1024-row chunk: its Nexus rows;
//   role_order    per chunk: the stable partition [ordinary rows | Nexus rows]
//                 (perm[g] = source row of grouped row g) and the two group
//                 sizes;
//   row_gather    the rows of X in grouped order (warp per row, 16-byte loads),
//                 except slabs of grouped rows that are runs of X's rows, which
//                 the GEMM loads from X directly;
//   routed_gemm   a persistent tcgen05 GEMM on CTA pairs over 256 x 256
//                 output tiles of the grouped rows.  A tile never straddles
//                 the two groups, so each tile reads one weight matrix; the
//                 epilogue writes bf16 rows to the parts.
#include "sonic_dev.cuh"
#include "sonic_host.h"

namespace sonic {
namespace {

constexpr int kChunkRows = 1024;  // rows per block of the partition kernels
constexpr int kGBM = 256;         // output tile rows (grouped rows) of a CTA pair
constexpr int kHalfM = 128;       // of them in each CTA
constexpr int kGBN = 256;         // output tile columns
constexpr int kHalfN = 128;       // weight rows each CTA stages
constexpr int kGBK = 64;          // reduction step (one 128-byte swizzle row)
constexpr int kGStages = 6;
constexpr int kGThreads = 192;    // warp 0 TMA, warp 1 MMA (leader), warps 2-5 epilogue
constexpr int kMaxParts = 4;

// ------------------------------------------------------------- partition

__global__ void __launch_bounds__(256)
role_count_kernel(const uint8_t *__restrict__ role, int32_t T, int32_t *__restrict__ counts) {
    const int c = blockIdx.x;
    int n = 0;
#pragma unroll
    for (int j = 0; j < kChunkRows / 256; ++j) {
        const int t = c * kChunkRows + j * 256 + threadIdx.x;
        n += (t < T && role[t] == SONIC_ROLE_NEXUS);
    }
    __shared__ int red[8];
    for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = n;
    __syncthreads();
    if (threadIdx.x == 0) {
        int s = 0;
        for (int w = 0; w < 8; ++w) s += red[w];
        counts[c] = s;
    }
}

// Thread = row.  Ordinary rows keep their order at the front, Nexus rows
// theirs after all ordinary rows.
__global__ void __launch_bounds__(kChunkRows)
role_order_kernel(const uint8_t *__restrict__ role, int32_t T, int32_t n_chunks,
                  const int32_t *__restrict__ counts, int32_t *__restrict__ perm,
                  int32_t *__restrict__ groups) {
    const int c = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    __shared__ int sh_before, sh_total;
    __shared__ int warp_tot[kChunkRows / 32];
    if (warp == 0) {
        int before = 0, total = 0;
        for (int i = lane; i < n_chunks; i += 32) {
            const int v = counts[i];
            total += v;
            if (i < c) before += v;
        }
        for (int o = 16; o > 0; o >>= 1) {
            before += __shfl_xor_sync(0xffffffffu, before, o);
            total += __shfl_xor_sync(0xffffffffu, total, o);
        }
        if (lane == 0) {
            sh_before = before;
            sh_total = total;
        }
    }
    const int t = c * kChunkRows + tid;
    const int nex = (t < T && role[t] == SONIC_ROLE_NEXUS) ? 1 : 0;
    int incl = nex;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += u;
    }
    if (lane == 31) warp_tot[warp] = incl;
    __syncthreads();
    int wbase = 0;
    for (int w = 0; w < warp; ++w) wbase += warp_tot[w];
    const int rank1 = wbase + incl - nex;  // Nexus rows before t in this chunk
    const int before = sh_before, n0 = T - sh_total;
    if (t < T) {
        const int g = nex ? n0 + before + rank1 : (c * kChunkRows - before) + (tid - rank1);
        perm[g] = t;
    }
    if (c == 0 && tid == 0) {
        groups[0] = n0;
        groups[1] = sh_total;
    }
}

// The GEMM stages A in slabs of 128 grouped rows, counted from the start of
// each role group (a CTA's share of a 256-row pair tile).  Grouped rows keep
// their order within a group, so a slab is one run of consecutive rows of X
// exactly when its first and last source rows are as far apart as its rows;
// the GEMM then loads the slab from X itself and it is not copied.
__device__ __forceinline__ int slab_start(int g, int n0) {
    return g < n0 ? (g / kHalfM) * kHalfM : n0 + ((g - n0) / kHalfM) * kHalfM;
}

__device__ __forceinline__ bool slab_is_run(const int32_t *perm, int s0, int group_end) {
    const int e = min(s0 + kHalfM, group_end);
    return perm[e - 1] - perm[s0] == e - 1 - s0;
}

// Xg[g] = X[perm[g]] for the rows of slabs that are not runs of X: one warp
// per row, 16-byte loads.
__global__ void __launch_bounds__(256)
row_gather_kernel(const uint8_t *__restrict__ X, int64_t x_row_bytes, int32_t T,
                  int64_t row_bytes, const int32_t *__restrict__ perm,
                  const int32_t *__restrict__ groups, uint8_t *__restrict__ Xg) {
    const int lane = threadIdx.x & 31;
    const int64_t n_warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int cpr = (int)(row_bytes >> 4);
    const int n0 = groups[0];
    for (int64_t g = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; g < T; g += n_warps) {
        if (slab_is_run(perm, slab_start((int)g, n0), g < n0 ? n0 : T)) continue;
        const uint8_t *src = X + (int64_t)perm[g] * x_row_bytes;
        uint8_t *dst = Xg + g * row_bytes;
        for (int c0 = lane; c0 < cpr; c0 += 128) {
            int4 v[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int c = c0 + 32 * u;
                if (c < cpr) v[u] = __ldg(reinterpret_cast<const int4 *>(src) + c);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int c = c0 + 32 * u;
                if (c < cpr) reinterpret_cast<int4 *>(dst)[c] = v[u];
            }
        }
    }
}

// ------------------------------------------------------------- GEMM
//
// The GEMM runs on CTA pairs (clusters of two) with the 2-SM form of the
// tensor-core MMA: a pair computes a 256 x 256 output tile, each CTA holding
// 128 rows of A and 128 of the tile's 256 weight rows, and the even CTA
// issues MMAs that read both CTAs' shared memory and write 128 accumulator
// rows into each CTA's tensor memory.  The 1-SM form with a 128 x 256 tile
// reads 96 B/clk of operands from shared memory while the TMA writes another
// 96 B/clk into it, more than shared memory delivers; the pair form halves
// the B traffic per SM.

struct GemmPart {
    uint16_t *base;
    int64_t stride;  // elements between rows
    int64_t rows;    // rows of base
    int col0, cols;
    int scatter;
};

struct GemmParams {
    const int32_t *groups;  // [2]: ordinary rows, Nexus rows
    const int32_t *perm;
    const int32_t *dst_row;
    GemmPart part[kMaxParts];
    int n_parts;
    int T, d_in, d_out, n_tiles_n;
    int32_t *status;
};

struct GemmCfg {
    static constexpr int kABytes = kHalfM * kGBK * 2;  // 16 KB: this CTA's 128 rows of A
    static constexpr int kBBytes = kHalfN * kGBK * 2;  // 16 KB: its 128 weight rows
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr int kOffBar = kGStages * kStageBytes;
    static constexpr int kNumBars = 2 * kGStages + 5;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;
    static constexpr size_t kSmem = 1024 + kOffMisc + 16;
};

// Tile i of the schedule: its grouped-row start, its valid-row end, its
// column tile and its weight matrix.  m runs fastest, so the pairs working
// at one time share the weight tiles of one column tile.
struct GemmTile {
    int row0, row_end, n, g;
};

__device__ __forceinline__ GemmTile gemm_tile(int i, int n0, int n1, int mt0, int total_m) {
    GemmTile w;
    const int m = i % total_m;
    w.n = i / total_m;
    if (m < mt0) {
        w.g = 0;
        w.row0 = m * kGBM;
        w.row_end = n0;
    } else {
        w.g = 1;
        w.row0 = n0 + (m - mt0) * kGBM;
        w.row_end = n0 + n1;
    }
    return w;
}

// After an abort, how long the non-leading CTA of a pair leaves its issued
// copies to land before it may exit (ns).
constexpr uint64_t kCopyGraceNs = 200000;

// ---- CTA-pair primitives (clusters of two CTAs; rank 0 leads)

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// Address of the same shared-memory offset in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t smem_in_rank(const void *p, uint32_t rank) {
    uint32_t a;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_u32(p)), "r"(rank));
    return a;
}

__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
                 : "memory");
}

// TMA load into this CTA's shared memory, completion counted on an mbarrier
// of either CTA of the pair: in the pair form, bit 24 of the barrier's
// shared-memory address selects the CTA, so the leader's barrier at the same
// offset is the address with that bit cleared.
__device__ __forceinline__ void tma_load_pair(void *dst, const CUtensorMap *map, uint32_t bar,
                                              int32_t c0, int32_t c1) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cta.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
        " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(0), "r"(0)
        : "memory");
}

__device__ __forceinline__ void tmem_alloc_pair(uint32_t *dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(dst_smem)),
                 "r"(ncols)
                 : "memory");
}

__device__ __forceinline__ void tmem_relinquish_pair() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}

__device__ __forceinline__ void mma_pair_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive once on the mbarrier at `bar`'s offset in every CTA of `mask` when
// the pair MMAs this thread issued so far are complete.
__device__ __forceinline__ void commit_pair(uint64_t *bar, uint16_t mask) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
        " [%0], %1;" ::"r"(smem_u32(bar)),
        "h"(mask)
        : "memory");
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGThreads, 1)
routed_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmX,
                   const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmWn,
                   const GemmParams p) {
    using C = GemmCfg;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + C::kOffBar);
    uint64_t *full = bars;                     // [stages] both CTAs' tiles landed (leader)
    uint64_t *empty = bars + kGStages;         // [stages] the MMAs reading them are done
    uint64_t *acc_full = bars + 2 * kGStages;  // [2] accumulator complete
    uint64_t *acc_empty = acc_full + 2;        // [2] read out by both CTAs (leader, 256)
    uint64_t *mma_idle = acc_empty + 2;
    int32_t *misc = reinterpret_cast<int32_t *>(smem + C::kOffMisc);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t rank = cluster_rank();
    const int cid = blockIdx.x >> 1, n_clusters = gridDim.x >> 1;
    // no early return: both CTAs of the pair must reach the cluster barriers
    const int n0 = p.groups[0], n1 = p.groups[1];
    const int mt0 = (n0 + kGBM - 1) / kGBM, mt1 = (n1 + kGBM - 1) / kGBM;
    const int total_m = mt0 + mt1;
    const int n_tiles = timed_out(p.status) ? 0 : total_m * p.n_tiles_n;
    const int nk = p.d_in / kGBK;

    if (tid == 0) {
        for (int s = 0; s < kGStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], 2 * 128);
        }
        mbar_init(mma_idle, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc_pair(reinterpret_cast<uint32_t *>(&misc[0]), 512);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync_all();  // both CTAs' barriers and tensor memory are set up
    tc_fence_after();
    const uint32_t tmem = static_cast<uint32_t>(misc[0]);

    int issued = 0;  // pipeline stages this CTA's producer filled (for the drain)
    if (warp == 0) {
        // ------------------------------------------------------------ producers
        // Each CTA loads its 128 rows of A and its 128 weight rows; both
        // count on the leader's `full` barrier, which the leader arms with
        // the pair's bytes.
        if (lane == 0) {
            tma_prefetch_desc(&tmA);
            tma_prefetch_desc(&tmX);
            tma_prefetch_desc(&tmW);
            tma_prefetch_desc(&tmWn);
            int it = 0;
            bool ok = true;
            for (int i = cid; ok && i < n_tiles; i += n_clusters) {
                const GemmTile w = gemm_tile(i, n0, n1, mt0, total_m);
                const CUtensorMap *tb = w.g ? &tmWn : &tmW;
                // this CTA's 128 rows of A: straight from X when they are one run
                // of X's rows, else from the grouped copy
                const int s0 = w.row0 + (int)rank * kHalfM;
                const bool run = s0 < w.row_end && slab_is_run(p.perm, s0, w.row_end);
                const CUtensorMap *ta = run ? &tmX : &tmA;
                const int arow = run ? p.perm[s0] : s0;
                for (int kb = 0; kb < nk; ++kb, ++it) {
                    const int s = it % kGStages;
                    if (it >= kGStages &&
                        !mbar_wait(&empty[s], ((it / kGStages) - 1) & 1, p.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    uint8_t *a = smem + s * C::kStageBytes;
                    if (rank == 0) mbar_arrive_expect_tx(&full[s], 2 * C::kStageBytes);
                    const uint32_t bar = smem_u32(&full[s]) & 0xFEFFFFFFu;
                    tma_load_pair(a, ta, bar, kb * kGBK, arow);
                    tma_load_pair(a + C::kABytes, tb, bar, kb * kGBK,
                                  w.n * kGBN + (int)rank * kHalfN);
                    issued = it + 1;
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer (leader)
        if (lane == 0 && rank == 0) {
            constexpr uint32_t idesc = idesc_bf16_f32(kGBM, kGBN, 0, 0);
            const uint32_t base = smem_u32(smem);
            int it = 0, j = 0;
            bool ok = true;
            for (int i = cid; ok && i < n_tiles; i += n_clusters, ++j) {
                const int b = j & 1;
                if (j >= 2 && !mbar_wait(&acc_empty[b], ((j >> 1) - 1) & 1, p.status, abort_flag))
                    break;
                tc_fence_after();
                const uint32_t acc = tmem + b * kGBN;
                for (int kb = 0; kb < nk; ++kb, ++it) {
                    const int s = it % kGStages;
                    if (!mbar_wait(&full[s], (it / kGStages) & 1, p.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a_addr = base + s * C::kStageBytes;
                    const uint32_t b_addr = a_addr + C::kABytes;
#pragma unroll
                    for (int kk = 0; kk < kGBK / 16; ++kk)
                        mma_pair_ss(acc, smem_desc_sw128(a_addr + kk * 32, 16, 1024),
                                    smem_desc_sw128(b_addr + kk * 32, 16, 1024), idesc,
                                    (kb > 0 || kk > 0) ? 1u : 0u);
                    commit_pair(&empty[s], 3);  // frees the stage in both CTAs
                }
                if (ok) commit_pair(&acc_full[b], 3);
            }
            // every MMA issued by this thread has finished once this arrives (a
            // wait bounded by time alone: the pair's memory is released after it)
            commit_pair(mma_idle, 1);
            mbar_drain(mma_idle, 0);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int quarter = warp & 3;
        const int r = quarter * 32 + lane;  // this CTA's tile row = TMEM lane
        const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
        int j = 0;
        for (int i = cid; i < n_tiles; i += n_clusters, ++j) {
            const int b = j & 1;
            const GemmTile w = gemm_tile(i, n0, n1, mt0, total_m);
            const int g = w.row0 + (int)rank * kHalfM + r;
            const bool valid = g < w.row_end;
            const int t = valid ? p.perm[g] : 0;
            const int dst = (valid && p.dst_row != nullptr) ? p.dst_row[t] : t;
            if (!mbar_wait(&acc_full[b], (j >> 1) & 1, p.status, abort_flag)) break;
            tc_fence_after();
#pragma unroll 1
            for (int c = 0; c < kGBN / 32; ++c) {
                const int col = w.n * kGBN + c * 32;
                if (col >= p.d_out) break;  // block-uniform
                uint32_t v[32];
                tmem_ld32(tmem + lane_base + b * kGBN + c * 32, v);
                tmem_ld_wait();
                reg_fence32(v);
                if (!valid) continue;
                // the part holding these 32 columns (parts are multiples of 32 wide)
                int k = 0;
#pragma unroll
                for (int q = 1; q < kMaxParts; ++q)
                    if (q < p.n_parts && col >= p.part[q].col0) k = q;
                const GemmPart &pt = p.part[k];
                const int64_t row = pt.scatter ? dst : t;
                if (row < 0 || row >= pt.rows) {  // outside the part: not written
                    set_status(p.status, SONIC_ERR_CAPACITY);
                    continue;
                }
                uint4 *out = reinterpret_cast<uint4 *>(pt.base + row * pt.stride + (col - pt.col0));
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    out[u] = make_uint4(
                        pack_bf16x2(__uint_as_float(v[8 * u + 0]), __uint_as_float(v[8 * u + 1])),
                        pack_bf16x2(__uint_as_float(v[8 * u + 2]), __uint_as_float(v[8 * u + 3])),
                        pack_bf16x2(__uint_as_float(v[8 * u + 4]), __uint_as_float(v[8 * u + 5])),
                        pack_bf16x2(__uint_as_float(v[8 * u + 6]), __uint_as_float(v[8 * u + 7])));
            }
            // this accumulator is read out: the MMAs of tile j + 2 may reuse it
            tc_fence_before();
            mbar_arrive_cluster(smem_in_rank(&acc_empty[b], 0));
        }
    }
    tc_fence_before();
    __syncthreads();
    // After an abort no thread of this CTA waits any more; let the copies in
    // flight land before the pair's memory goes away.  Both CTAs' copies of a
    // stage complete on the leader's barrier, so the leader drains the stages
    // it armed; the other CTA cannot wait on that barrier and gives its own
    // copies a bounded grace period instead (a copy that is issued lands in
    // microseconds).
    if (*abort_flag && warp == 0 && lane == 0) {
        if (rank == 0) {
            for (int u = max(0, issued - kGStages); u < issued; ++u)
                mbar_drain(&full[u % kGStages], (u / kGStages) & 1);
        } else if (issued > 0) {
            const uint64_t t0 = global_ns();
            while (global_ns() - t0 < kCopyGraceNs) __nanosleep(1000);
        }
    }
    __syncthreads();
    cluster_sync_all();  // no CTA leaves while its pair may still touch its memory
    tc_fence_after();
    if (warp == 1) tmem_dealloc_pair(tmem, 512);
}

struct RlWorkspace {
    size_t counts, groups, perm, xg, total;
};

RlWorkspace rl_workspace(const sonic_routed_linear_args *a) {
    RlWorkspace w{};
    const size_t T = a->n_rows > 0 ? (size_t)a->n_rows : 0;
    const size_t chunks = (T + kChunkRows - 1) / kChunkRows;
    w.counts = 0;
    w.groups = round_up(chunks * 4, 256);
    w.perm = w.groups + 256;
    w.xg = w.perm + round_up(T * 4, 256);
    w.total = w.xg + round_up(T * (size_t)(a->d_in > 0 ? a->d_in : 0) * 2, 256);
    return w;
}

}  // namespace
}  // namespace sonic

using namespace sonic;

extern "C" size_t sonic_routed_linear_workspace_size(const sonic_routed_linear_args *a) {
    if (a == nullptr || a->n_rows <= 0 || a->d_in <= 0) return 0;
    return rl_workspace(a).total;
}

extern "C" sonic_status_t sonic_routed_linear(const uint16_t *X, const uint16_t *W,
                                              const uint16_t *W_nexus, const uint8_t *role,
                                              const sonic_routed_linear_args *a,
                                              sonic_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (a == nullptr || a->n_rows < 0) return SONIC_ERR_INVALID_ARGUMENT;
    if (a->n_rows == 0) return SONIC_OK;
    if (X == nullptr || W == nullptr || W_nexus == nullptr || role == nullptr)
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->d_in <= 0 || a->d_in % kGBK != 0 || a->d_out <= 0 || a->d_out % 32 != 0)
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->x_row_stride < a->d_in || a->x_row_stride % 8 != 0) return SONIC_ERR_INVALID_ARGUMENT;
    if (!aligned16(X) || !aligned16(W) || !aligned16(W_nexus)) return SONIC_ERR_INVALID_ARGUMENT;
    if (a->n_parts < 1 || a->n_parts > kMaxParts) return SONIC_ERR_INVALID_ARGUMENT;
    GemmParams p{};
    int col = 0;
    for (int k = 0; k < a->n_parts; ++k) {
        const sonic_out_part &q = a->parts[k];
        if (q.base == nullptr || !aligned16(q.base) || q.cols <= 0 || q.cols % 32 != 0 ||
            q.row_stride < q.cols || q.row_stride % 8 != 0 || q.rows <= 0)
            return SONIC_ERR_INVALID_ARGUMENT;
        if (q.scatter && a->dst_row == nullptr) return SONIC_ERR_INVALID_ARGUMENT;
        if (!q.scatter && q.rows < a->n_rows) return SONIC_ERR_INVALID_ARGUMENT;
        p.part[k] = GemmPart{static_cast<uint16_t *>(q.base), q.row_stride, q.rows, col, q.cols,
                             q.scatter ? 1 : 0};
        col += q.cols;
    }
    if (col != a->d_out) return SONIC_ERR_INVALID_ARGUMENT;
    if ((long long)a->n_rows * a->d_in > (1LL << 40)) return SONIC_ERR_UNSUPPORTED;
    const RlWorkspace ws = rl_workspace(a);
    if (a->workspace == nullptr || a->workspace_bytes < ws.total) return SONIC_ERR_WORKSPACE;

    char *wsb = static_cast<char *>(a->workspace);
    int32_t *counts = reinterpret_cast<int32_t *>(wsb + ws.counts);
    int32_t *groups = reinterpret_cast<int32_t *>(wsb + ws.groups);
    int32_t *perm = reinterpret_cast<int32_t *>(wsb + ws.perm);
    uint16_t *Xg = reinterpret_cast<uint16_t *>(wsb + ws.xg);
    const int T = a->n_rows;
    const int chunks = (T + kChunkRows - 1) / kChunkRows;

    // tensor maps: grouped rows of X, and the two weight matrices
    const uint64_t adims[4] = {(uint64_t)a->d_in, (uint64_t)T, 1, 1};
    const uint64_t astr[3] = {(uint64_t)a->d_in * 2, (uint64_t)a->d_in * 2 * T,
                              (uint64_t)a->d_in * 2 * T};
    // boxes: one CTA's share of a stage (128 rows of A, 128 weight rows)
    const uint32_t abox[4] = {kGBK, kHalfM, 1, 1};
    const uint64_t wdims[4] = {(uint64_t)a->d_in, (uint64_t)a->d_out, 1, 1};
    const uint64_t wstr[3] = {(uint64_t)a->d_in * 2, (uint64_t)a->d_in * 2 * a->d_out,
                              (uint64_t)a->d_in * 2 * a->d_out};
    const uint32_t wbox[4] = {kGBK, kHalfN, 1, 1};
    static_assert(kGBK * kHalfM * 2 == GemmCfg::kABytes && kGBK * kHalfN * 2 == GemmCfg::kBBytes,
                  "TMA boxes must fill exactly one stage slot");
    // X itself, for slabs of grouped rows that are runs of X's rows
    const uint64_t xdims[4] = {(uint64_t)a->d_in, (uint64_t)T, 1, 1};
    const uint64_t xstr[3] = {(uint64_t)a->x_row_stride * 2, (uint64_t)a->x_row_stride * 2 * T,
                              (uint64_t)a->x_row_stride * 2 * T};
    CUtensorMap tA, tX, tW, tWn;
    if (!make_tmap_bf16_4d(&tA, Xg, adims, astr, abox) ||
        !make_tmap_bf16_4d(&tX, X, xdims, xstr, abox) ||
        !make_tmap_bf16_4d(&tW, W, wdims, wstr, wbox) ||
        !make_tmap_bf16_4d(&tWn, W_nexus, wdims, wstr, wbox))
        return SONIC_ERR_INVALID_ARGUMENT;

    role_count_kernel<<<chunks, 256, 0, stream>>>(role, T, counts);
    role_order_kernel<<<chunks, kChunkRows, 0, stream>>>(role, T, chunks, counts, perm, groups);
    const int sms = device_sm_count();
    const long long gwarps = (long long)sms * 8 * 8;  // 8 blocks of 8 warps per SM at most
    const int gblocks = (int)((T < gwarps ? T : gwarps) + 7) / 8;
    row_gather_kernel<<<gblocks, 256, 0, stream>>>(
        reinterpret_cast<const uint8_t *>(X), a->x_row_stride * 2, T, (int64_t)a->d_in * 2, perm,
        groups, reinterpret_cast<uint8_t *>(Xg));

    p.groups = groups;
    p.perm = perm;
    p.dst_row = a->dst_row;
    p.n_parts = a->n_parts;
    p.T = T;
    p.d_in = a->d_in;
    p.d_out = a->d_out;
    p.n_tiles_n = (a->d_out + kGBN - 1) / kGBN;
    p.status = a->status;
    const long long max_tiles = ((long long)(T + kGBM - 1) / kGBM + 1) * p.n_tiles_n;
    const int pairs = (int)(max_tiles < sms / 2 ? max_tiles : sms / 2);
    const int blocks = 2 * (pairs > 0 ? pairs : 1);
    constexpr size_t smem = GemmCfg::kSmem;
    static_assert(smem <= 232448, "routed GEMM shared memory");
    cudaError_t e = cudaFuncSetAttribute(routed_gemm_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return SONIC_ERR_CUDA;
    routed_gemm_kernel<<<blocks, kGThreads, smem, stream>>>(tA, tX, tW, tWn, p);
    return cudaGetLastError() == cudaSuccess ? SONIC_OK : SONIC_ERR_CUDA;
}
