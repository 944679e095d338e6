/*
 * sonic.h -- C ABI of libsonic, the GB300 (sm_103a) attention path over a
 * Nexus-compressed KV cache (SONIC, arXiv 2601.21927).
 *
 * Three operations, in the order a dialogue goes through them:
 *
 *   sonic_compact_kv    keep only the system-prompt, Nexus and current-turn
 *                       K/V rows of every sequence and layer (the retention
 *                       rule: Sec. 1, the Fig. 2 caption, Sec. 3.2 "Historical
 *                       Body Removal", App. C effective context I_sys + N + Q_n).
 *   sonic_attn_prefill  softmax attention of a sequence's query rows under the
 *                       hierarchical visibility mask of Sec. 3.2 (Eq. 3 causal
 *                       rule, Eq. 4 body removal, Eq. 5 bidirectional Nexus).
 *   sonic_attn_decode   one generation step with grouped-query heads over the
 *                       retained cache (App. C, Eq. 15: generation conditions
 *                       on I_sys, the Nexus state and the current query only).
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Every tensor and metadata pointer is a DEVICE pointer owned by the
 *    caller.  The library never allocates, frees or synchronises; each call
 *    enqueues kernels on `stream` (a cudaStream_t; NULL is the legacy default
 *    stream) and returns.  Scratch memory comes from the caller's
 *    `workspace` (query its size first).
 *  - Host-detectable errors (NULL where a pointer is required, bad sizes,
 *    unsupported head_dim or head ratio, workspace too small, misaligned
 *    pointers) return a status before anything is launched.  Conditions only
 *    the GPU can see (output capacity exceeded, an inconsistent layout, a
 *    bounded wait that ran out) are written to the optional device word
 *    `*status` (first error wins; the caller zeroes it) and the affected
 *    blocks stop early; nothing traps.  sonic_read_status() fetches it.
 *  - Roles are per-token uint8 values (sonic_role_t); segment numbers are
 *    int32 (0 = system prompt, i = history segment m_i, h+1 = current turn,
 *    non-decreasing along a sequence).  Positions p, q of the mask are row
 *    numbers within one sequence, in S_aug order (Eq. 1).
 *  - Token rows of K and V hold all KV heads: element (row t, head j, dim d)
 *    sits at t * n_heads_kv * head_dim + j * head_dim + d.  Query rows hold
 *    all query heads the same way.  Query head h reads KV head
 *    h / (n_heads_q / n_heads_kv).
 *  - Attention tensors are bf16 (stored as uint16 bit patterns), accumulate
 *    in fp32 and write bf16 outputs rounded to nearest even.
 *  - Calls are stateless and may be issued from several host threads.
 */
#ifndef SONIC_H
#define SONIC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SONIC_ABI_VERSION 4

#if defined(__GNUC__)
#define SONIC_API __attribute__((visibility("default")))
#else
#define SONIC_API
#endif

/* cudaStream_t without including the CUDA headers. */
typedef struct CUstream_st *sonic_stream_t;

/* Per-token role in the augmented sequence S_aug (Sec. 3.1, Eq. 1). */
typedef enum {
    SONIC_ROLE_SYS = 0,   /* system prompt I_sys                     */
    SONIC_ROLE_BODY = 1,  /* text of a history segment, B_i          */
    SONIC_ROLE_NEXUS = 2, /* Nexus token of a history segment, N_i   */
    SONIC_ROLE_CURR = 3   /* current query / current turn, Q_curr    */
} sonic_role_t;

typedef enum {
    SONIC_OK = 0,
    SONIC_ERR_INVALID_ARGUMENT = 1,
    SONIC_ERR_UNSUPPORTED = 2,
    SONIC_ERR_WORKSPACE = 3,
    SONIC_ERR_CAPACITY = 4,
    SONIC_ERR_DEVICE_TIMEOUT = 5,
    SONIC_ERR_CUDA = 6,
    SONIC_ERR_LAYOUT = 7
} sonic_status_t;

/* Which Nexus tokens a Nexus token sees (Eq. 5 and its reading).
 * FULL: every Nexus token of every segment (Eq. 5 as printed).
 * CAUSAL_SEGMENTS: Nexus tokens of its own and earlier segments only (the
 * reading under which Nexus state is kept across a session, Sec. 6.4).
 * Rows that are not Nexus tokens see the same keys under both. */
typedef enum {
    SONIC_NEXUS_FULL = 0,
    SONIC_NEXUS_CAUSAL_SEGMENTS = 1
} sonic_nexus_vis_t;

/* Order in which sonic_attn_prefill walks a sequence's keys (and queries).
 * AS_GIVEN: the key rows as laid out (S_aug order).
 * RETAINED_FIRST: the library first lays each sequence's keys out in its
 * workspace (role, segment, position) as [system prompt, Nexus and
 * current-turn rows | history bodies], each part in S_aug order and the
 * bodies starting on a 128-row boundary; the mask still compares S_aug
 * positions.  Every query row then sees one prefix of the retained part plus
 * (for body and Nexus rows) the body of its own segment, so far fewer key
 * tiles are visited and cut by the mask when all rows of S_aug are queried.
 * A 128-key tile of that order made of 128 consecutive rows of K and V (a
 * stretch of one body, of the system prompt or of the current turn) is read
 * from K and V in place; the K and V rows of every other tile are copied into
 * the workspace, for every layer.  Unless query heads are packed (short query
 * blocks), the query rows are walked in the same order too, by 32-row chunks
 * of runs (one body, or consecutive rows that are not body rows), so a query
 * tile holds rows that see nearly the same keys; Q and O stay where they are.
 * A sequence with more than 1024 such runs, or whose runs padded to 32 rows
 * exceed align128(q_len) + 1024 rows, keeps the given query order.  Results
 * equal AS_GIVEN up to floating-point summation order.  The layout and the
 * copies cost workspace: see sonic_prefill_workspace_size. */
typedef enum {
    SONIC_KEYS_AS_GIVEN = 0,
    SONIC_KEYS_RETAINED_FIRST = 1
} sonic_key_order_t;

/* ------------------------------------------------------------------------- */
/* Compaction                                                                */
/* ------------------------------------------------------------------------- */

typedef struct {
    int32_t batch;               /* B >= 0 sequences                                    */
    int32_t n_layers;            /* >= 1; K/V of every layer are compacted in one call  */
    const int32_t *k_start;      /* device [B]: first packed row of sequence b           */
    const int32_t *k_len;        /* device [B]: rows of sequence b (raw S_aug length)    */
    const int32_t *reserve;      /* device [B] or NULL: free rows left after sequence
                                    b's retained rows (room to append new tokens)       */
    int64_t row_bytes;           /* bytes of one token row (all KV heads); multiple of 16 */
    int64_t in_layer_bytes;      /* byte stride between layers of K and V; multiple of 16 */
    int64_t out_layer_bytes;     /* byte stride between layers of out_K and out_V       */
    int32_t out_capacity_rows;   /* rows available per layer in out_K / out_V           */
    int32_t *ret_len;            /* device [B] or NULL: retained rows of sequence b      */
    int32_t *src_idx;            /* device [out_capacity_rows] or NULL: packed source row
                                    of each output row, -1 in reserve rows              */
    uint8_t *out_role;           /* device [out_capacity_rows] or NULL: role of each
                                    output row (SONIC_ROLE_BODY in reserve rows)        */
    int32_t *out_seg;            /* device [out_capacity_rows] or NULL: segment of each
                                    output row (-1 in reserve rows)                     */
    int32_t *status;             /* device int32 or NULL                                */
    void *workspace;             /* device, sonic_compact_workspace_size() bytes        */
    size_t workspace_bytes;
    int32_t total_rows;          /* rows per layer of K, V, role, seg_id (> 0); a
                                    sequence outside them is refused                    */
} sonic_compact_args;

/*
 * Retention rule (Sec. 3.2 body removal; App. C effective context): row t of
 * sequence b is kept iff role[t] != SONIC_ROLE_BODY.  Kept rows keep their
 * order.  Writes
 *   offsets[b] = sum_{b' < b} (ret_len[b'] + reserve[b'])  (device [B+1],
 *                offsets[B] = total output rows),
 * and for every layer l and kept row j of sequence b copies the row_bytes of
 * K (resp. V) row k_start[b] + (j-th kept position) of layer l to row
 * offsets[b] + j of layer l of out_K (resp. out_V), bit for bit.  Reserve
 * rows are not written.  seg_id may be NULL; when given it is checked
 * (non-decreasing within a sequence, no body row in segment 0) and a
 * violation sets SONIC_ERR_LAYOUT.  If offsets[B] > out_capacity_rows the
 * call sets SONIC_ERR_CAPACITY and copies only rows below the capacity.
 * K/V/out pointers must be 16-byte aligned.  B > 65535 or n_layers > 32767
 * returns SONIC_ERR_UNSUPPORTED.  A sequence whose rows fall outside
 * [0, total_rows) keeps no rows (ret_len 0) and sets
 * SONIC_ERR_INVALID_ARGUMENT in *status; none of its rows is read.
 */
SONIC_API sonic_status_t sonic_compact_kv(const void *K, const void *V, const int32_t *seg_id,
                                const uint8_t *role, void *out_K, void *out_V,
                                int32_t *offsets, const sonic_compact_args *args,
                                sonic_stream_t stream);

/* Workspace bytes sonic_compact_kv needs for these args (0 if none). */
SONIC_API size_t sonic_compact_workspace_size(const sonic_compact_args *args);

/* ------------------------------------------------------------------------- */
/* Masked prefill                                                            */
/* ------------------------------------------------------------------------- */

typedef struct {
    int32_t batch;               /* B >= 0                                              */
    int32_t n_layers;            /* >= 1                                                */
    int32_t n_heads_q;           /* Hq, a multiple of n_heads_kv                        */
    int32_t n_heads_kv;          /* Hkv >= 1                                            */
    int32_t head_dim;            /* D: 64 or 128                                        */
    const int32_t *k_start;      /* device [B]: first key row of sequence b in K, V,
                                    role, seg_id                                        */
    const int32_t *k_len;        /* device [B]: key rows of sequence b                   */
    const int32_t *q_start;      /* device [B]: first query row of sequence b in Q, O    */
    const int32_t *q_len;        /* device [B]: query rows of sequence b, <= k_len[b];
                                    query i is key position k_len[b] - q_len[b] + i
                                    (the last q_len rows: bottom-right aligned)         */
    int32_t max_q_len;           /* host: >= every q_len[b]; sizes the launch grid      */
    int32_t max_k_len;           /* host: >= every k_len[b], at most 262144 (262016
                                    with key_order RETAINED_FIRST)                      */
    int32_t total_q_rows;        /* rows per layer of Q and O                           */
    int32_t total_k_rows;        /* rows per layer of K and V (and of role, seg_id)     */
    int64_t q_layer_stride;      /* elements between layers of Q                        */
    int64_t kv_layer_stride;     /* elements between layers of K and V                  */
    int64_t o_layer_stride;      /* elements between layers of O                        */
    float softmax_scale;         /* 0 selects 1/sqrt(head_dim)                          */
    int32_t nexus_vis;           /* sonic_nexus_vis_t                                   */
    float *lse;                  /* device [n_layers][total_q_rows][Hq] or NULL: natural
                                    log-sum-exp of each row's scaled visible scores     */
    int32_t *status;             /* device int32 or NULL                                */
    void *workspace;             /* device, sonic_prefill_workspace_size() bytes        */
    size_t workspace_bytes;
    int32_t key_order;           /* sonic_key_order_t                                   */
    float *nexus_mass;           /* device [n_layers][total_q_rows][Hq] or NULL: share of
                                    each row's attention on visible Nexus keys          */
} sonic_prefill_args;

/*
 * Sec. 3.2 masked attention.  For every layer, sequence b, query row i and
 * query head h, with p = k_len[b] - q_len[b] + i:
 *   s_q   = scale * <Q[p, h], K[q, h/G]>  for the key rows q of sequence b,
 *   vis   = the Sec. 3.2 rule on (role, seg_id) of rows p and q:
 *             key q a body row:           same segment and q <= p   (Eqs. 3, 4)
 *             both Nexus rows:            true (FULL) or seg[q] <= seg[p]   (Eq. 5)
 *             otherwise:                  q <= p                    (Eq. 3)
 *   O[i, h] = sum_{q in vis} softmax(s)_q V[q, h/G]   (zeros if nothing is visible).
 * Whole 128x128 key tiles the mask hides are skipped; the rule is applied per
 * element only on tiles it cuts.  Q, K, V, O are bf16; every row stride and
 * base pointer must be 16-byte aligned.  role and seg_id are indexed like the
 * key rows of one layer (shared by all layers); role 255 marks a row that is
 * no key (padding).  key_order picks the order the key tiles are cut in
 * (sonic_key_order_t).  A sequence with q_len[b] > k_len[b], k_len[b] >
 * max_k_len, or rows outside [0, total_k_rows) / [0, total_q_rows) is refused
 * with SONIC_ERR_INVALID_ARGUMENT in *status (none of its rows is read).
 * nexus_mass (optional) is the per-row, per-head quantity behind A_nexus of
 * the Nexus attention regularisation (Sec. 4.1, Eq. 9):
 *   nexus_mass[i, h] = sum_{q in vis, role[q] = NEXUS} softmax(s)_q
 * (0 when nothing is visible), normalised like O, i.e. over the bf16-rounded
 * probabilities the P.V product uses.  The paper's A_nexus is its mean over
 * heads and current-turn rows, a reduction left to the caller.
 */
SONIC_API sonic_status_t sonic_attn_prefill(const uint16_t *Q, const uint16_t *K, const uint16_t *V,
                                  const int32_t *seg_id, const uint8_t *role, uint16_t *O,
                                  const sonic_prefill_args *args, sonic_stream_t stream);

/*
 * Workspace bytes for sonic_attn_prefill with these arguments (0 for an empty
 * batch).  AS_GIVEN: 256 bytes for the counter the persistent blocks claim
 * work units from, then 32 + 256 bytes per 128-key tile (its summary and its
 * column masks), batch * ceil(max_k_len / 128) tiles, each part rounded up to
 * 256 bytes.  RETAINED_FIRST counts one more tile per sequence and adds 4
 * bytes per tile, batch * (align128(max_q_len) + 1024) / 8 bytes (the query
 * order's chunk table) and, for R = min(batch * (align128(max_k_len) + 128),
 * total_k_rows + 256 * batch) rows: 13 bytes of metadata per row and a K and
 * a V copy of R rows for every layer (2 * n_layers * R * n_heads_kv *
 * head_dim * 2 bytes).  Sequence b takes align128(k_len[b]) + 128 of the R
 * rows; sequences that share key rows can need more than R, which the GPU
 * reports as SONIC_ERR_WORKSPACE in *status.
 */
SONIC_API size_t sonic_prefill_workspace_size(const sonic_prefill_args *args);

/*
 * sonic_attn_prefill for callers that cannot allocate device memory.  The
 * paper has no counterpart; this is a deployment aid.  Some callers cannot
 * call cudaMalloc: code running inside a custom allocator or memory-pool
 * callback, runtimes that plan every device byte ahead of time, or hosts that
 * only hand over fixed buffers for inputs and outputs.  This call takes the
 * same arguments as sonic_attn_prefill except that args->workspace and
 * args->workspace_bytes are ignored: the per-tile summaries and column masks
 * live in a fixed array of 9 MiB + 256 bytes compiled into the library
 * (every GPU that loads the library holds it until the process exits).  It
 * allocates nothing.
 *  - Limit: batch * ceil(max_k_len / 128) <= 32768; larger calls return
 *    SONIC_ERR_WORKSPACE before launching anything.  Only key_order AS_GIVEN
 *    is served (RETAINED_FIRST copies K and V into the workspace):
 *    SONIC_ERR_UNSUPPORTED otherwise.
 *  - The first call on each device looks up the array's device address
 *    (cudaGetSymbolAddress, with that device current) and caches it with the
 *    id of the device's current context; make that first call before any
 *    stream capture.  After a device reset the context id differs, so the
 *    next call looks the address up again (make it outside a capture too).
 *  - Every call on a device shares the one array and leaves its contents
 *    behind; each call rewrites every entry it reads, so nothing needs
 *    clearing, but calls that overlap on the GPU (other streams, other host
 *    threads) race on it and must be serialised by the caller.
 */
SONIC_API sonic_status_t sonic_attn_prefill_static(const uint16_t *Q, const uint16_t *K,
                                                   const uint16_t *V, const int32_t *seg_id,
                                                   const uint8_t *role, uint16_t *O,
                                                   const sonic_prefill_args *args,
                                                   sonic_stream_t stream);

/* ------------------------------------------------------------------------- */
/* Decode                                                                    */
/* ------------------------------------------------------------------------- */

typedef struct {
    int32_t batch;               /* B >= 0                                              */
    int32_t n_layers;            /* >= 1; all layers run in one launch                  */
    int32_t n_heads_q;           /* Hq, a multiple of n_heads_kv, Hq / Hkv <= 16        */
    int32_t n_heads_kv;          /* Hkv >= 1                                            */
    int32_t head_dim;            /* D: 64 or 128                                        */
    const int32_t *kv_start;     /* device [B]: first retained row of sequence b         */
    int32_t max_len;             /* host: >= every lens[b]; sizes the split grid        */
    int32_t total_kv_rows;       /* rows per layer of K_ret and V_ret                   */
    int64_t q_layer_stride;      /* elements between layers of q                        */
    int64_t kv_layer_stride;     /* elements between layers of K_ret and V_ret          */
    int64_t o_layer_stride;      /* elements between layers of O                        */
    float softmax_scale;         /* 0 selects 1/sqrt(head_dim)                          */
    int32_t chunk_len;           /* keys per split (0 = automatic), rounded up to the key
                                    tile of 128 keys                                    */
    float *lse;                  /* device [n_layers][B][Hq] or NULL                    */
    int32_t *status;             /* device int32 or NULL                                */
    void *workspace;             /* device, sonic_decode_workspace_size() bytes         */
    size_t workspace_bytes;
    const uint8_t *role;         /* device [total_kv_rows] or NULL: role of each retained
                                    row (needed for nexus_mass)                         */
    float *nexus_mass;           /* device [n_layers][B][Hq] or NULL: share of the
                                    attention on rows whose role is SONIC_ROLE_NEXUS    */
} sonic_decode_args;

/*
 * One decode step (App. C).  q and O are [n_layers][B][Hq][D] (layer strides
 * given); for sequence b the retained rows kv_start[b] .. kv_start[b] +
 * lens[b] - 1 of K_ret / V_ret (the new token's own row included) are all
 * visible:  O[l, b, h] = sum_t softmax_t(scale <q[l,b,h], K[t, h/G]>) V[t, h/G].
 * The keys are split into chunks of chunk_len; each (layer, sequence, KV
 * head, chunk) unit produces a partial (max, sum, accumulator) in the
 * workspace, and a second kernel merges them by log-sum-exp (a sequence that
 * fits one chunk is written directly).  One persistent block per SM claims
 * units from a counter in the workspace (zeroed on `stream` before the
 * launch), so the workspace is never empty and concurrent calls need
 * workspaces of their own.  A sequence whose rows fall outside [0, total_kv_rows) is
 * refused with SONIC_ERR_INVALID_ARGUMENT in *status (its outputs are left
 * undefined).  lens[b] = 0 gives zeros (and
 * lse = -inf).  bf16 in/out, fp32 arithmetic.  nexus_mass (optional, role
 * then required, else SONIC_ERR_INVALID_ARGUMENT) is the decode form of the
 * quantity behind A_nexus (Sec. 4.1, Eq. 9): the share of the new token's
 * attention, per query head, on retained rows t with role[kv_start[b] + t]
 * = SONIC_ROLE_NEXUS (0 when lens[b] = 0); it adds one float per (unit,
 * chunk) to the workspace.
 */
SONIC_API sonic_status_t sonic_attn_decode(const uint16_t *q, const uint16_t *K_ret,
                                 const uint16_t *V_ret, const int32_t *lens, uint16_t *O,
                                 const sonic_decode_args *args, sonic_stream_t stream);

SONIC_API size_t sonic_decode_workspace_size(const sonic_decode_args *args);

/* ------------------------------------------------------------------------- */
/* Role-routed projections                                                   */
/* ------------------------------------------------------------------------- */

/* One output part: a range of `cols` consecutive columns of Y (the parts
 * take Y's columns in order), written as bf16 rows of `base`. */
typedef struct {
    void *base;                  /* device bf16, 16-byte aligned                         */
    int64_t row_stride;          /* elements between rows of base; multiple of 8, >= cols */
    int32_t cols;                /* > 0, multiple of 32                                 */
    int32_t scatter;             /* 0: row t of Y goes to row t; 1: to row dst_row[t]   */
    int64_t rows;                /* rows of base: a row index outside [0, rows) is not
                                    written and sets SONIC_ERR_CAPACITY in *status      */
} sonic_out_part;

typedef struct {
    int32_t n_rows;              /* T >= 0 rows (tokens) of X                           */
    int32_t d_in;                /* columns of X and of W: a multiple of 64             */
    int32_t d_out;               /* rows of W = the parts' columns together; multiple of 32 */
    int64_t x_row_stride;        /* elements between rows of X; multiple of 8, >= d_in  */
    const int32_t *dst_row;      /* device [T] or NULL (required if a part scatters)    */
    int32_t n_parts;             /* 1 .. 4                                              */
    sonic_out_part parts[4];
    int32_t *status;             /* device int32 or NULL                                */
    void *workspace;             /* device, sonic_routed_linear_workspace_size() bytes  */
    size_t workspace_bytes;
} sonic_routed_linear_args;

/*
 * Role-routed linear map (Sec. 3.1: Nexus tokens have their own projection
 * matrices W_Q^N, W_K^N, W_V^N, W_O^N):
 *   Y[t, n] = sum_k X[t, k] * Wsel(t)[n, k],
 *   Wsel(t) = W_nexus if role[t] == SONIC_ROLE_NEXUS, W otherwise,
 * X [T][x_row_stride] bf16 (the first d_in columns used), W and W_nexus
 * [d_out][d_in] bf16 contiguous (a linear layer's out x in layout; W_nexus
 * may equal W), fp32 accumulation, Y rounded to bf16 (nearest even) and
 * written part by part.  For a QKV projection the parts are Q (row t of the
 * query buffer) and K and V (row dst_row[t] of this layer's K and V caches:
 * the rows compaction reserved), so new tokens' keys and values land in the
 * retained cache with no further copy.  Rows are grouped by role on the GPU
 * (a stable partition, no host round trip) and the GEMM runs on the tensor
 * cores; the workspace holds the grouped copy of X.  T = 0 does nothing.
 */
SONIC_API sonic_status_t sonic_routed_linear(const uint16_t *X, const uint16_t *W,
                                             const uint16_t *W_nexus, const uint8_t *role,
                                             const sonic_routed_linear_args *args,
                                             sonic_stream_t stream);

/* Workspace bytes for sonic_routed_linear: about T * (d_in * 2 + 4) bytes. */
SONIC_API size_t sonic_routed_linear_workspace_size(const sonic_routed_linear_args *args);

/* ------------------------------------------------------------------------- */
/* Status                                                                    */
/* ------------------------------------------------------------------------- */

/* Waits for `stream`, then copies the device status word to the host and
 * returns it (SONIC_ERR_CUDA if the copy itself fails). */
SONIC_API sonic_status_t sonic_read_status(const int32_t *status, sonic_stream_t stream);

/* Static, human-readable name of a status code. */
SONIC_API const char *sonic_status_string(sonic_status_t status);

/* SONIC_ABI_VERSION of the loaded library. */
SONIC_API int32_t sonic_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SONIC_H */
