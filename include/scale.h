/*
 * scale.h -- C ABI of libscale, a GB300 (sm_103a) implementation of the
 * prefill hot path of Similarity Chunk Rolling (SCR), the long-context engine
 * of SCALE (arXiv 2609.31568, Sec. V-A).
 *
 * SCR runs chunked prefill with selective sparse attention (Sec. III-B, Def. 1,
 * Eq. 3-4) and performs the selection once per *cluster* of similar query
 * sub-chunks instead of once per sub-chunk (Algorithm 2). The path has four
 * steps, exposed as three calls:
 *
 *   scale_build_reps      (a) block representative keys, sub-chunk
 *                             fingerprints (Eq. 6) and anchor-based clusters
 *                             (Eq. 8, Algorithm 1); scale_build_reps_range
 *                             does the same chunk by chunk;
 *   scale_select          (b) GQA-aware scoring of the representatives against
 *                             each cluster's anchor fingerprint with head
 *                             soft-voting, and (c) a deterministic top-k
 *                             (Eq. 9, Sec. V-A3 "Selection function
 *                             instantiation");
 *   scale_sparse_prefill  (d) block-sparse causal attention over sinks,
 *                             selected blocks and the cluster-spanning local
 *                             window with an online softmax (Eq. 10).
 *
 * SCALE_MODE_PER_SUBCHUNK runs the same steps with every sub-chunk as its own
 * unit: the per-sub-chunk (TokenSelect-style) baseline of Sec. III-A.
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Layouts. Q and O: bf16 [N][H_q][d_h]; K and V: bf16 [N][H_kv][d_h]
 *    (token-major, head_dim innermost, contiguous). Query head h reads KV head
 *    h / (H_q / H_kv). Representatives: fp32 [H_kv][nb][d_h], nb = ceil(N/B).
 *    Fingerprints: fp32 [M][H_q*d_h], M = ceil(N/L). Unit table: int32
 *    unit_start[M+1], unit u covering sub-chunks [unit_start[u],
 *    unit_start[u+1]), plus a device int32 n_units. Selection: int32
 *    sel_blocks[M][top_k] (ascending, -1 padded) and int32 sel_count[M],
 *    row u = unit u.
 *  - Pointers. All data pointers are DEVICE pointers (except where a name says
 *    _host), 16-byte aligned, owned by the caller. The library allocates no
 *    memory on any path; scratch lives in a caller-provided workspace of
 *    scale_workspace_size() bytes, initialised once with scale_workspace_init().
 *    (scale_prefill_host creates, for the duration of the call, two streams
 *    and their events to overlap its copies with the compute.)
 *  - Streams. `stream` is a cudaStream_t (NULL = legacy default stream). Calls
 *    only enqueue work on it and never synchronise, except the functions
 *    documented as synchronous (scale_get_device_status, scale_prefill_host).
 *  - Errors. Argument problems are reported synchronously by the return value
 *    (scale_status_t); nothing is enqueued then. Device-side problems (a
 *    bounded wait that ran out, a failed bounds check) are recorded in a status
 *    word inside the workspace and read with scale_get_device_status(). There
 *    is no CPU fallback: every step runs in this library's CUDA kernels.
 *  - Concurrency. Calls are reentrant; two calls that share a workspace must
 *    not overlap on the GPU.
 *  - Supported shapes: head_dim 128, H_q / H_kv at most 32 (at most 8 for
 *    token-level selection and decode), H_kv at most 64, N < 2^31,
 *    outer_chunk a multiple of sub_chunk.
 */
#ifndef SCALE_H
#define SCALE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A cudaStream_t; declared here so that the header needs no CUDA include. */
typedef struct CUstream_st *scale_stream_t;

typedef enum {
    SCALE_OK = 0,
    SCALE_ERR_INVALID_ARG = -1, /* a null/misaligned pointer or inconsistent sizes */
    SCALE_ERR_UNSUPPORTED = -2, /* valid but outside what the kernels implement */
    SCALE_ERR_WORKSPACE = -3,   /* workspace smaller than scale_workspace_size() */
    SCALE_ERR_CUDA = -4,        /* a CUDA runtime call failed */
    SCALE_ERR_TIMEOUT = -5,     /* device status: a bounded wait ran out */
    SCALE_ERR_DEVICE = -6       /* device status: a device-side check failed */
} scale_status_t;

typedef enum {
    SCALE_MODE_PER_CLUSTER = 0,  /* SCR: one selection per cluster (Algorithm 2) */
    SCALE_MODE_PER_SUBCHUNK = 1  /* baseline: one selection per sub-chunk (Sec. III-A) */
} scale_mode_t;

/* Problem description. Notation of the paper in brackets. */
typedef struct scale_params {
    int32_t num_q_heads;           /* [H]  query heads                                   */
    int32_t num_kv_heads;          /*      KV heads; divides num_q_heads (GQA)           */
    int32_t head_dim;              /* [d_h] must be 128                                  */
    int32_t sub_chunk;             /* [L]  sub-chunk length in tokens                    */
    int64_t n_tokens;              /* [N]  tokens of Q, K and V                          */
    int32_t max_cluster_subchunks; /* [L_max / L] cluster cap (Eq. 8)                    */
    int32_t outer_chunk;           /* [L_outer] tokens; 0 means L_max; multiple of L     */
    float theta;                   /* [theta] admission threshold (Eq. 8);
                                      <= -1 admits every sub-chunk                       */
    int32_t block_size;            /* [B]  KV block size of the selection, tokens        */
    int32_t top_k;                 /* [k]  selected blocks per unit                      */
    int32_t n_sink;                /* [n_init] leading sink tokens always attended       */
    int32_t n_local;               /* [n_local^base] window before the unit's first token */
    float select_scale;            /* sigma: logit scale inside the per-head softmax     */
    float attn_scale;              /* softmax scale of Eq. 10; 0 means 1/sqrt(d_h)       */
} scale_params_t;

/* Bytes of workspace that scale_build_reps / scale_select / scale_sparse_prefill
 * need for `p` and `mode` (one workspace serves all three). Synchronous, host only. */
int scale_workspace_size(const scale_params_t *p, int32_t mode, size_t *bytes);

/* Zero the workspace header (the device status word). Call once after
 * allocating a workspace, and again to clear a recorded device error. */
int scale_workspace_init(void *ws, size_t ws_bytes, scale_stream_t stream);

/* Step (a). Eq. 6 and Sec. V-A1: fingerprints[i] = mean of the multi-head
 * queries of sub-chunk i (tokens [iL, min(N,(i+1)L))); block representative
 * key of block b and KV head j = mean of K over the tokens of the block;
 * Algorithm 1 with the admission rule of Eq. 8 inside each outer chunk of
 * outer_chunk tokens, producing unit_start[0..n_units] (entries after
 * n_units are set to M) and *n_units (device).
 *   q            bf16 [N][H_q][128]        k  bf16 [N][H_kv][128]
 *   reps         fp32 [H_kv][nb][128]      out (may be NULL when block_size is 1)
 *   fingerprints fp32 [M][H_q*128]         out (raw means v_i, not normalised)
 *   unit_start   int32 [M+1]               out
 *   n_units      int32 [1]                 out (device)
 */
int scale_build_reps(const scale_params_t *p, const void *q, const void *k, float *reps,
                     float *fingerprints, int32_t *unit_start, int32_t *n_units, void *ws,
                     size_t ws_bytes, scale_stream_t stream);

/* Step (a) over the outer chunks that cover tokens [tok_begin, tok_end), for a
 * caller that prefills chunk by chunk (Sec. III-B) and has the rows of later
 * chunks not yet on the device. tok_begin is a multiple of the outer chunk
 * length L_outer; tok_end is one too, or N. The ranges of a sequence are
 * issued in order on one stream, starting at 0 and without gaps: each call
 * appends its units to unit_start after the *n_units units of the earlier
 * ranges (the first range, tok_begin = 0, starts the table), so that after the
 * range ending at N the outputs equal those of scale_build_reps bit for bit.
 * A call reads Q rows [tok_begin, tok_end) and K rows [tok_begin - B + 1,
 * tok_end); it writes the fingerprints of the range's sub-chunks and the
 * representatives of the blocks whose last token lies in the range (the range
 * ending at N also writes the final, partial block). Arguments and errors as
 * for scale_build_reps; a range that breaks the rules above returns
 * SCALE_ERR_INVALID_ARG, and tok_begin == tok_end enqueues nothing. */
int scale_build_reps_range(const scale_params_t *p, int64_t tok_begin, int64_t tok_end, const void *q,
                           const void *k, float *reps, float *fingerprints, int32_t *unit_start,
                           int32_t *n_units, void *ws, size_t ws_bytes, scale_stream_t stream);

/* Step (a) without a workspace. The paper has no counterpart: this entry point
 * exists for callers that cannot allocate device memory for the library, such
 * as a host framework's plugin interface that hands over only input and output
 * buffers, or a serving loop whose device memory pool is fully reserved and
 * where a cudaMalloc (which may synchronise the device) is not allowed on the
 * request path. It computes exactly what scale_build_reps computes, with the
 * same arguments minus the workspace, and allocates nothing: its scratch is a
 * fixed 16 MiB array inside the library, which every GPU that loads the
 * library holds until the process exits.
 *  - Limit: returns SCALE_ERR_WORKSPACE, without launching anything, when the
 *    scratch step (a) needs for `p` exceeds 16 MiB (it grows with
 *    M * (ceil(H_q / 2) + max_cluster_subchunks + 1) * 4 bytes plus 256; 34 KB
 *    for 1M tokens with L = 4096, about 34 MB, which is rejected, for 128M
 *    tokens with L = 512).
 *  - Set-up: the first call on each device looks up the array's device address
 *    with that device current; make that first call before any stream capture.
 *  - Sharing: every call on a device uses the same array, which keeps the last
 *    call's contents (step (a) writes each scratch element before reading it,
 *    so nothing is cleared between calls); calls whose work overlaps on the
 *    GPU (other streams, or other host threads) race on it and must be
 *    serialised by the caller.
 *  - Errors: argument checks as for scale_build_reps, returned synchronously.
 *    There is no device status to read: step (a)'s kernels have no bounded
 *    waits or device-side checks and record none. */
int scale_build_reps_noalloc(const scale_params_t *p, const void *q, const void *k, float *reps,
                             float *fingerprints, int32_t *unit_start, int32_t *n_units,
                             scale_stream_t stream);

/* Steps (b) and (c). Eq. 9 with head soft-voting (Sec. V-A3): for every unit u
 * starting in [tok_begin, tok_end) (SCR: the clusters of unit_start; baseline:
 * the sub-chunks) with anchor sub-chunk a (its first), and every query head h:
 *   z_{h,b} = select_scale * v_a^(h) . r_b^(h / g)
 * over the candidate blocks b that hold a token in [n_sink, W_u),
 * W_u = max(0, s_u - n_local); p_h = softmax_b(z_h); score_b = sum_h p_{h,b};
 * the top_k blocks by (score descending, block index ascending), written to
 * sel_blocks[u] in ascending order, -1 padded; sel_count[u] = min(top_k,
 * |candidates|). tok_begin and tok_end must be multiples of outer_chunk (SCR)
 * or sub_chunk (baseline), or tok_end == N.
 *   sel_scores  fp32 [M][nb] or NULL: score_b on the candidates, NaN elsewhere.
 * unit_start / n_units are ignored in baseline mode (may be NULL). */
int scale_select(const scale_params_t *p, int32_t mode, int64_t tok_begin, int64_t tok_end,
                 const float *reps, const float *fingerprints, const int32_t *unit_start,
                 const int32_t *n_units, int32_t *sel_blocks, int32_t *sel_count,
                 float *sel_scores, void *ws, size_t ws_bytes, scale_stream_t stream);

/* Steps (b) and (c) at token granularity (block_size must be 1): the rule of
 * scale_select with every key as its own block, which is the paper's own
 * selection (Sec. V-A3, Eq. 9, TokenSelect's head soft-voting over tokens):
 *   z_{h,t} = select_scale * v_a^(h) . k_t^(h / g)  for n_sink <= t < W_u,
 *   p_h = softmax_t(z_h), score_t = sum_h p_{h,t}, top_k tokens (ties to the
 *   lower index), ascending.
 * The scores are computed from K directly on the tensor cores (the fp32
 * fingerprint split into three bf16 parts, fp32 accumulation), so
 * scale_build_reps may be given reps = NULL for block size 1.
 *   k           bf16 [N][H_kv][128]
 *   sel_tokens  int32 [M][top_k] out (ascending token indices, -1 padded)
 *   sel_count   int32 [M] out
 *   sel_scores  fp32 [M][N] or NULL: score_t on the candidates, NaN elsewhere.
 * Same range rule, modes and workspace as scale_select. H_q / H_kv must be at
 * most 8 (SCALE_ERR_UNSUPPORTED otherwise); block_size != 1 gives
 * SCALE_ERR_INVALID_ARG (and scale_select gives SCALE_ERR_UNSUPPORTED for
 * block size 1). */
int scale_select_tokens(const scale_params_t *p, int32_t mode, int64_t tok_begin, int64_t tok_end,
                        const void *k, const float *fingerprints, const int32_t *unit_start,
                        const int32_t *n_units, int32_t *sel_tokens, int32_t *sel_count,
                        float *sel_scores, void *ws, size_t ws_bytes, scale_stream_t stream);

/* Step (d). Eq. 10 for every query row p of every unit u starting in
 * [tok_begin, tok_end) and every query head h:
 *   keys K(p) = ([0, n_sink) U selected blocks of u U [W_u, e_u)) n [0, p],
 *   taken as a set (each key once), with W_u = max(0, s_u - n_local);
 *   out[p][h] = sum_{t in K(p)} softmax_t(attn_scale * q_p^(h) . k_t^(h/g)) v_t^(h/g)
 * computed with bf16 tensor-core products, fp32 accumulation and an online
 * softmax; probabilities are rounded to bf16 before the product with V; out
 * is rounded to bf16 (nearest even). Rows outside [tok_begin, tok_end) are
 * not written. Same range rule as scale_select.
 *   q, out bf16 [N][H_q][128];  k, v bf16 [N][H_kv][128];
 *   sel_blocks / sel_count as written by scale_select (any selection obeying
 *   the same layout is accepted; entries outside [0, nb) are ignored). With
 *   block_size 1 they are scale_select_tokens' token lists, and the kernel
 *   gathers the selected keys and values row by row (entries outside
 *   [n_sink, W_u) or not above their predecessor are ignored). */
int scale_sparse_prefill(const scale_params_t *p, int32_t mode, int64_t tok_begin,
                         int64_t tok_end, const void *q, const void *k, const void *v,
                         const int32_t *unit_start, const int32_t *n_units,
                         const int32_t *sel_blocks, const int32_t *sel_count, void *out,
                         void *ws, size_t ws_bytes, scale_stream_t stream);

/* Paged KV cache (the serving layout, as paged attention engines keep it):
 * K and V live in a pool of num_pages pages of page_size tokens,
 *   k_pages, v_pages  bf16 [num_pages][page_size][H_kv][128]  (device)
 * and token t of the sequence is row t % page_size of page
 * page_table[t / page_size] (int32, device, ceil(N / page_size) entries).
 * The *_paged entry points below compute exactly what their contiguous
 * counterparts compute (bit for bit, for the same K and V values).
 *  - Every K/V box the kernels load is 64 rows starting at a multiple of 64,
 *    so page_size, sub_chunk, n_sink and n_local must be multiples of 64 and
 *    block_size 1 or a multiple of 64 (SCALE_ERR_UNSUPPORTED otherwise), and
 *    num_pages * page_size < 2^31.
 *  - A page-table entry outside [0, num_pages) is not dereferenced: its
 *    tokens read as zero keys and values. Q and the attention output stay
 *    contiguous.
 *  - The rows of the last page past token N - 1 are loaded with their box and
 *    masked out (weight exactly 0); they must hold finite values (zeros, or
 *    any data), since 0 times a NaN would still be NaN. */
typedef struct {
    const void *k_pages;
    const void *v_pages;
    const int32_t *page_table;
    int32_t page_size;
    int64_t num_pages;
} scale_kv_pages_t;

/* scale_build_reps with K read from a paged cache. */
int scale_build_reps_paged(const scale_params_t *p, const void *q, const scale_kv_pages_t *kv,
                           float *reps, float *fingerprints, int32_t *unit_start, int32_t *n_units,
                           void *ws, size_t ws_bytes, scale_stream_t stream);

/* scale_build_reps_range with K read from a paged cache. */
int scale_build_reps_range_paged(const scale_params_t *p, int64_t tok_begin, int64_t tok_end, const void *q,
                                 const scale_kv_pages_t *kv, float *reps, float *fingerprints,
                                 int32_t *unit_start, int32_t *n_units, void *ws, size_t ws_bytes,
                                 scale_stream_t stream);

/* scale_select_tokens with K read from a paged cache. */
int scale_select_tokens_paged(const scale_params_t *p, int32_t mode, int64_t tok_begin,
                              int64_t tok_end, const scale_kv_pages_t *kv, const float *fingerprints,
                              const int32_t *unit_start, const int32_t *n_units, int32_t *sel_tokens,
                              int32_t *sel_count, float *sel_scores, void *ws, size_t ws_bytes,
                              scale_stream_t stream);

/* scale_sparse_prefill with K and V read from a paged cache. */
int scale_sparse_prefill_paged(const scale_params_t *p, int32_t mode, int64_t tok_begin,
                               int64_t tok_end, const void *q, const scale_kv_pages_t *kv,
                               const int32_t *unit_start, const int32_t *n_units,
                               const int32_t *sel_blocks, const int32_t *sel_count, void *out,
                               void *ws, size_t ws_bytes, scale_stream_t stream);

/* One decode step with a selection cache. The paper's method targets prefill
 * and leaves decode to its engine, whose selection cache reuses a token
 * selection across consecutive, highly similar decode queries (Sec. VII).
 * This step applies the paper's rules with one query token (Def. 1, C = 1):
 *  - the query q_t of position t (its K and V rows already at row t) is the
 *    unit's fingerprint; its candidates are the tokens n_sink <= c < W_t,
 *    W_t = max(0, t - n_local);
 *  - reuse: with an anchor in `cache`, the step reuses the anchor's selection
 *    when cos(q_t, anchor) >= theta (all heads together, as Eq. 8; a zero norm
 *    gives cosine 0) and fewer than max_cluster_subchunks steps have shared
 *    it; otherwise it retrieves (Eq. 9 at block size 1: per-head softmax over
 *    the candidates, head soft-vote, top_k tokens, ties to the lower index)
 *    and q_t becomes the anchor;
 *  - out_t[h] = Eq. 10 for the single row t over sinks U selection U [W_t, t].
 * Parameters: n_tokens = rows of k and v (t < n_tokens), block_size must be
 * 1, H_q / H_kv at most 8, H_q at most 96; sub_chunk and outer_chunk are not
 * used. The reuse decision is made on the device: a step never synchronises.
 *   q_t, out_t  bf16 [H_q][128];  k, v  bf16 [n_tokens][H_kv][128]
 *   cache       scale_decode_cache_size() bytes, zeroed by
 *               scale_decode_cache_init() before the first step of a sequence
 *   ws          scale_decode_workspace_size() bytes (grows with n_tokens); its
 *               first 256 bytes hold the device status word: zero them once
 *               with scale_workspace_init(); a bounded wait of the step that
 *               runs out records SCALE_ERR_TIMEOUT there, read with
 *               scale_get_device_status(). */
int scale_decode_cache_size(const scale_params_t *p, size_t *bytes);
int scale_decode_cache_init(void *cache, size_t cache_bytes, scale_stream_t stream);
int scale_decode_workspace_size(const scale_params_t *p, size_t *bytes);
int scale_decode_step(const scale_params_t *p, int64_t t, const void *q_t, const void *k, const void *v,
                      void *cache, size_t cache_bytes, void *out_t, void *ws, size_t ws_bytes,
                      scale_stream_t stream);

/* Synchronous: waits for `stream`, then reads the device status word of `ws`
 * into *status (SCALE_OK, SCALE_ERR_TIMEOUT or SCALE_ERR_DEVICE). The word is
 * sticky until scale_workspace_init(). */
int scale_get_device_status(const void *ws, scale_stream_t stream, int32_t *status);

/* Host-only bookkeeping of the cost model of Sec. V-A2: given a unit table in
 * HOST memory, the number of units and how many of them make a retrieval call
 * (non-empty candidate set). Baseline mode ignores unit_start_host. */
int scale_retrieval_calls(const scale_params_t *p, int32_t mode, const int32_t *unit_start_host,
                          int32_t n_units, int64_t *units, int64_t *calls);

/* End to end from HOST buffers: copies q, k, v (host, bf16 layouts above) to
 * the device, runs steps (a)-(d) over all tokens, copies the attention output
 * back to out_host, and waits for `stream`. `arena` is a caller-owned device
 * buffer of scale_prefill_host_arena_size() bytes that holds the device copies,
 * the intermediate tensors and the workspace. Host buffers may be pageable;
 * pinned buffers make the copies asynchronous with respect to the host.
 * The call runs as chunked prefill does (Sec. III-B): in pieces of whole outer
 * chunks (at most 64 pieces), each computed with the range calls
 * (scale_build_reps_range, scale_select, scale_sparse_prefill) once its rows
 * have arrived, while the next piece's rows are copied in and the previous
 * piece's output is copied out on two streams of the call's own. When L or
 * n_local is not a multiple of 128 it runs as one piece. The result equals the
 * whole-sequence calls bit for bit. The call creates and releases those
 * streams and their events itself. */
int scale_prefill_host_arena_size(const scale_params_t *p, int32_t mode, size_t *bytes);
int scale_prefill_host(const scale_params_t *p, int32_t mode, const void *q_host,
                       const void *k_host, const void *v_host, void *out_host, void *arena,
                       size_t arena_bytes, scale_stream_t stream);

/* Upper bound, in nanoseconds of wall time, of every device-side wait of the
 * attention kernel (default 4e9). A wait that runs out records
 * SCALE_ERR_TIMEOUT in the device status and the kernel returns. Process-wide;
 * applies to launches issued after the call. ns = 0 is refused with
 * SCALE_ERR_INVALID_ARG and leaves the limit unchanged. */
int scale_set_wait_timeout_ns(uint64_t ns);

/* Self-check of the bounded-wait machinery: launches one block that waits on an
 * mbarrier nothing arrives at, with a limit of `timeout_ns`; the kernel records
 * SCALE_ERR_TIMEOUT in the device status of `ws` and returns. */
int scale_selftest_wait_timeout(void *ws, size_t ws_bytes, uint64_t timeout_ns,
                                scale_stream_t stream);

const char *scale_status_string(int status);

/* Library ABI version (major * 10000 + minor * 100 + patch). */
int scale_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SCALE_H */
