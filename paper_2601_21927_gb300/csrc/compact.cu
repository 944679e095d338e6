// KV compaction: keep the system-prompt, Nexus and current-turn rows of every
// sequence and layer, drop the history bodies.
//
// Retention rule (SONIC Sec. 3.2 "Historical Body Removal" and App. C: the
// effective context is I_sys + Nexus state + current query): a row is kept
// iff its role is not BODY; kept rows keep their order.
//
// Four launches, none of which needs a host round trip:
//   keep_count    one block per (chunk, sequence), each sequence cut into
//                 kChunks pieces: kept rows of the piece (and a layout check
//                 when segment numbers are given);
//   keep_bases    one block: per-sequence totals and their exclusive scan
//                 (with the reserve rows) -> offsets, ret_len, capacity check;
//   keep_scatter  one block per (chunk, sequence): its output base (the
//                 sequence's offset plus the pieces before it), then a block
//                 prefix scan of the keep flags from warp-shuffle scans,
//                 writing the source row of every output row (-1 in reserve
//                 rows);
//   kv_gather     all layers, K and V: 16-byte vector copy of every kept row
//                 to its output row, grid-stride over rows of each layer.
#include "sonic_dev.cuh"
#include "sonic_host.h"

namespace sonic {
namespace {

constexpr int kScanThreads = 512;
constexpr int kChunks = 64;  // pieces per sequence in the scans

// Rows of sequence (start, len), or 0 when they fall outside [0, total): such a
// sequence is refused, keeps nothing and is never read.
__device__ __forceinline__ int32_t seq_rows(int32_t start, int32_t len, int32_t total) {
    return (start < 0 || len < 0 || (int64_t)start + len > total) ? 0 : len;
}

// Rows [*lo, *hi) of piece c of a sequence of len rows (32-row aligned pieces).
__device__ __forceinline__ void piece(int32_t len, int c, int32_t *lo, int32_t *hi) {
    const long long ch = (((long long)len + kChunks - 1) / kChunks + 31) & ~31LL;
    *lo = (int32_t)min((long long)len, c * ch);
    *hi = (int32_t)min((long long)len, (c + 1) * ch);
}

__global__ void __launch_bounds__(kScanThreads)
keep_count_kernel(const uint8_t *__restrict__ role, const int32_t *__restrict__ seg,
                  const int32_t *__restrict__ k_start, const int32_t *__restrict__ k_len,
                  int32_t total, int32_t *__restrict__ counts, int32_t *status) {
    const int c = blockIdx.x, b = blockIdx.y;
    const int32_t start = k_start[b];
    const int32_t len = seq_rows(start, k_len[b], total);
    if (c == 0 && threadIdx.x == 0 && len != k_len[b]) set_status(status, SONIC_ERR_INVALID_ARGUMENT);
    int32_t lo, hi;
    piece(len, c, &lo, &hi);
    int n = 0;
    bool bad = false;
    for (int32_t t = lo + threadIdx.x; t < hi; t += blockDim.x) {
        uint8_t r = role[start + t];
        n += (r != SONIC_ROLE_BODY);
        bad |= (r > SONIC_ROLE_CURR);
        if (seg != nullptr) {
            int32_t sv = seg[start + t];
            bad |= (r == SONIC_ROLE_BODY && sv <= 0);
            if (t > 0) bad |= (sv < seg[start + t - 1]);
        }
    }
    // block reduction
    __shared__ int red[kScanThreads / 32];
    __shared__ int bad_any;
    if (threadIdx.x == 0) bad_any = 0;
    __syncthreads();
    for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = n;
    if (bad) bad_any = 1;
    __syncthreads();
    if (threadIdx.x == 0) {
        int sum = 0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) sum += red[w];
        counts[b * kChunks + c] = sum;
        if (bad_any) set_status(status, SONIC_ERR_LAYOUT);
    }
}

// Inclusive warp scan of v (warp-shuffle).
__device__ __forceinline__ int warp_inclusive_scan(int v) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int u = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += u;
    }
    return v;
}

// Exclusive scan over the sequences of (kept rows + reserve): one block.
__global__ void __launch_bounds__(kScanThreads)
keep_bases_kernel(const int32_t *__restrict__ counts, const int32_t *__restrict__ reserve,
                  int32_t B, int32_t capacity, long long *__restrict__ seq_base,
                  int32_t *__restrict__ offsets, int32_t *__restrict__ ret_len,
                  int32_t *status) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr int kWarps = kScanThreads / 32;
    __shared__ long long warp_tot[kWarps];
    long long running = 0;
    for (int32_t b0 = 0; b0 < B; b0 += blockDim.x) {
        const int32_t b = b0 + tid;
        long long v = 0;
        int32_t kept = 0;
        if (b < B) {
            for (int c = 0; c < kChunks; ++c) kept += counts[b * kChunks + c];
            v = (long long)kept + (reserve ? reserve[b] : 0);
        }
        // inclusive warp scan of v
        long long incl = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            long long u = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += u;
        }
        if (lane == 31) warp_tot[warp] = incl;
        __syncthreads();
        long long wb = 0, tot = 0;
        for (int w = 0; w < kWarps; ++w) {
            if (w < warp) wb += warp_tot[w];
            tot += warp_tot[w];
        }
        if (b < B) {
            const long long base = running + wb + incl - v;
            seq_base[b] = base;
            offsets[b] = (int32_t)base;
            if (ret_len) ret_len[b] = kept;
        }
        running += tot;
        __syncthreads();
    }
    if (tid == 0) {
        offsets[B] = (int32_t)running;
        if (running > capacity || running > 0x7fffffffLL) set_status(status, SONIC_ERR_CAPACITY);
    }
}

__global__ void __launch_bounds__(kScanThreads)
keep_scatter_kernel(const uint8_t *__restrict__ role, const int32_t *__restrict__ seg,
                    const int32_t *__restrict__ k_start, const int32_t *__restrict__ k_len,
                    const int32_t *__restrict__ reserve, const int32_t *__restrict__ counts,
                    const long long *__restrict__ seq_base, int32_t capacity, int32_t total,
                    int32_t *__restrict__ src_idx, uint8_t *__restrict__ out_role,
                    int32_t *__restrict__ out_seg) {
    const int c = blockIdx.x, b = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr int kWarps = kScanThreads / 32;
    __shared__ int warp_tot[kWarps];
    // output base of this piece: the sequence's offset plus the earlier pieces
    long long base = seq_base[b];
    for (int i = 0; i < c; ++i) base += counts[b * kChunks + i];
    const int32_t start = k_start[b], len = seq_rows(start, k_len[b], total);
    int32_t lo, hi;
    piece(len, c, &lo, &hi);
    long long running = base;
    for (int32_t c0 = lo; c0 < hi; c0 += blockDim.x) {
        const int32_t t = c0 + tid;
        const int keep = (t < hi) && (role[start + t] != SONIC_ROLE_BODY);
        int incl = warp_inclusive_scan(keep);
        if (lane == 31) warp_tot[warp] = incl;
        __syncthreads();
        int warp_base = 0, chunk_tot = 0;
        for (int w = 0; w < kWarps; ++w) {
            int v = warp_tot[w];
            if (w < warp) warp_base += v;
            chunk_tot += v;
        }
        const long long o = running + warp_base + incl - keep;
        if (keep && o < capacity) {
            if (src_idx) src_idx[o] = start + t;
            if (out_role) out_role[o] = role[start + t];
            if (out_seg) out_seg[o] = seg ? seg[start + t] : 0;
        }
        running += chunk_tot;
        __syncthreads();
    }
    // Reserve rows (piece 0 writes them): no source.
    if (c == 0 && reserve != nullptr) {
        long long kept = 0;
        for (int i = 0; i < kChunks; ++i) kept += counts[b * kChunks + i];
        const int32_t res = reserve[b];
        for (int32_t r = tid; r < res; r += blockDim.x) {
            const long long o = seq_base[b] + kept + r;
            if (o < capacity) {
                if (src_idx) src_idx[o] = -1;
                if (out_role) out_role[o] = SONIC_ROLE_BODY;
                if (out_seg) out_seg[o] = -1;
            }
        }
    }
}

// 16-byte vector copy of kept rows.  blockIdx.y = layer * 2 + (0: K, 1: V).
// One warp copies whole rows (lane j takes 16-byte chunks j, j+32, ...); each
// warp works on two rows at a time with all their loads issued before the
// stores, so up to 8 x 16 bytes per thread are in flight.
constexpr int kGatherThreads = 256;


__device__ __forceinline__ int4 ld_stream(const void *p) {
    int4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.s32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// kGatherRows rows a warp moves per pass, kGatherUnroll 16-byte pieces of each
// per lane per step: 2 x 4 for rows under 2 KB, 4 x 2 for larger rows (more
// rows in flight helps the long rows; at 1 KB it measured slower).
template <int kGatherRows, int kGatherUnroll>
__global__ void __launch_bounds__(kGatherThreads)
kv_gather_kernel(const uint8_t *__restrict__ K, const uint8_t *__restrict__ V,
                 uint8_t *__restrict__ out_K, uint8_t *__restrict__ out_V,
                 const int32_t *__restrict__ offsets, const int32_t *__restrict__ src_idx,
                 int32_t B, int32_t capacity, int64_t row_bytes, int64_t in_layer_bytes,
                 int64_t out_layer_bytes) {
    const int layer = blockIdx.y >> 1;
    const bool is_v = blockIdx.y & 1;
    const uint8_t *src = (is_v ? V : K) + (int64_t)layer * in_layer_bytes;
    uint8_t *dst = (is_v ? out_V : out_K) + (int64_t)layer * out_layer_bytes;
    int64_t n_rows = offsets[B];
    if (n_rows > capacity) n_rows = capacity;
    const int lane = threadIdx.x & 31;
    const int64_t n_warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int cpr = (int)(row_bytes >> 4);  // 16-byte chunks per row
    // each warp moves kGatherRows rows per pass (n_warps apart), every lane
    // holding its 16-byte pieces of all of them in flight
    for (int64_t r0 = (((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5); r0 < n_rows;
         r0 += kGatherRows * n_warps) {
        int32_t sr[kGatherRows];
#pragma unroll
        for (int k = 0; k < kGatherRows; ++k) {
            const int64_t r = r0 + k * n_warps;
            sr[k] = r < n_rows ? src_idx[r] : -1;
        }
        for (int c0 = lane; c0 < cpr; c0 += 32 * kGatherUnroll) {
            int4 v[kGatherRows][kGatherUnroll];
#pragma unroll
            for (int k = 0; k < kGatherRows; ++k)
#pragma unroll
                for (int u = 0; u < kGatherUnroll; ++u) {
                    const int c = c0 + 32 * u;
                    if (c < cpr && sr[k] >= 0)
                        v[k][u] = ld_stream(src + (int64_t)sr[k] * row_bytes + ((int64_t)c << 4));
                }
#pragma unroll
            for (int k = 0; k < kGatherRows; ++k)
#pragma unroll
                for (int u = 0; u < kGatherUnroll; ++u) {
                    const int c = c0 + 32 * u;
                    if (c < cpr && sr[k] >= 0)
                        *reinterpret_cast<int4 *>(dst + (r0 + k * n_warps) * row_bytes +
                                                  ((int64_t)c << 4)) = v[k][u];
                }
        }
    }
}

}  // namespace
}  // namespace sonic

using namespace sonic;

extern "C" size_t sonic_compact_workspace_size(const sonic_compact_args *a) {
    if (a == nullptr || a->batch < 0) return 0;
    // per-piece counts, then per-sequence 64-bit bases, then (if the caller
    // gives no src_idx) the source row of every output row
    size_t ws = round_up((size_t)a->batch * kChunks * sizeof(int32_t), 256) +
                round_up((size_t)a->batch * sizeof(long long), 256);
    if (a->src_idx == nullptr)
        ws += round_up((size_t)(a->out_capacity_rows > 0 ? a->out_capacity_rows : 0) *
                           sizeof(int32_t),
                       256);
    return ws;
}

extern "C" sonic_status_t sonic_compact_kv(const void *K, const void *V, const int32_t *seg_id,
                                           const uint8_t *role, void *out_K, void *out_V,
                                           int32_t *offsets, const sonic_compact_args *a,
                                           sonic_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (a == nullptr || offsets == nullptr) return SONIC_ERR_INVALID_ARGUMENT;
    if (a->batch < 0 || a->n_layers < 1 || a->out_capacity_rows < 0)
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->batch == 0) {
        if (cudaMemsetAsync(offsets, 0, sizeof(int32_t), stream) != cudaSuccess)
            return SONIC_ERR_CUDA;
        return SONIC_OK;
    }
    if (K == nullptr || V == nullptr || role == nullptr || out_K == nullptr ||
        out_V == nullptr || a->k_start == nullptr || a->k_len == nullptr)
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->row_bytes <= 0 || (a->row_bytes & 15) || (a->in_layer_bytes & 15) ||
        (a->out_layer_bytes & 15))
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->n_layers > 1 && (a->in_layer_bytes <= 0 || a->out_layer_bytes <= 0))
        return SONIC_ERR_INVALID_ARGUMENT;
    if (!aligned16(K) || !aligned16(V) || !aligned16(out_K) || !aligned16(out_V))
        return SONIC_ERR_INVALID_ARGUMENT;
    if (a->n_layers > 32767 || a->batch > 65535) return SONIC_ERR_UNSUPPORTED;
    if (a->total_rows <= 0) return SONIC_ERR_INVALID_ARGUMENT;
    const size_t need = sonic_compact_workspace_size(a);
    if (need > 0 && (a->workspace == nullptr || a->workspace_bytes < need))
        return SONIC_ERR_WORKSPACE;

    char *ws = static_cast<char *>(a->workspace);
    int32_t *counts = reinterpret_cast<int32_t *>(ws);
    ws += round_up((size_t)a->batch * kChunks * sizeof(int32_t), 256);
    long long *seq_base = reinterpret_cast<long long *>(ws);
    ws += round_up((size_t)a->batch * sizeof(long long), 256);
    int32_t *src_idx = a->src_idx != nullptr ? a->src_idx : reinterpret_cast<int32_t *>(ws);

    const dim3 pieces(kChunks, a->batch);
    keep_count_kernel<<<pieces, kScanThreads, 0, stream>>>(role, seg_id, a->k_start, a->k_len,
                                                          a->total_rows, counts, a->status);
    keep_bases_kernel<<<1, kScanThreads, 0, stream>>>(counts, a->reserve, a->batch,
                                                      a->out_capacity_rows, seq_base, offsets,
                                                      a->ret_len, a->status);
    keep_scatter_kernel<<<pieces, kScanThreads, 0, stream>>>(
        role, seg_id, a->k_start, a->k_len, a->reserve, counts, seq_base, a->out_capacity_rows,
        a->total_rows, src_idx, a->out_role, a->out_seg);
    const int sms = device_sm_count();
    // ~32 blocks per SM in all (four resident at a time): with many small
    // blocks the SMs run out of work together, where ~8 left a ragged tail
    // (5.9 -> 6.7 TB/s on a 28-layer compaction of 1 KB rows).
    const int per_slice = (sms * 32 + 2 * a->n_layers - 1) / (2 * a->n_layers);
    dim3 grid(per_slice < 1 ? 1 : per_slice, 2 * a->n_layers);
    auto gather = a->row_bytes >= 2048 ? kv_gather_kernel<4, 2> : kv_gather_kernel<2, 4>;
    gather<<<grid, kGatherThreads, 0, stream>>>(
        static_cast<const uint8_t *>(K), static_cast<const uint8_t *>(V),
        static_cast<uint8_t *>(out_K), static_cast<uint8_t *>(out_V), offsets, src_idx, a->batch,
        a->out_capacity_rows, a->row_bytes, a->in_layer_bytes, a->out_layer_bytes);
    return cudaGetLastError() == cudaSuccess ? SONIC_OK : SONIC_ERR_CUDA;
}
