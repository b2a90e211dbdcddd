// scale_internal.h -- definitions shared by the library's translation units:
// derived sizes, workspace layout, launch helpers of the kernels and the
// device-side unit table.
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "../../include/scale.h"

namespace scale {

constexpr int kHeadDim = 128;
constexpr int kSegRows = 64;         // rows of one K/V TMA box (a "segment")
constexpr int kMaxSegments = 1024;   // distant segments per unit the attention kernel can hold
constexpr int kStatusOffset = 0;     // device status word (int32) at the start of the workspace
constexpr size_t kAlign = 256;

// Device status word values: 0, SCALE_ERR_TIMEOUT, SCALE_ERR_DEVICE.

struct Derived {
    int64_t N;
    int Hq, Hkv, g, dh;
    int L;           // sub-chunk
    int S_max;       // max sub-chunks per cluster
    int per_outer;   // sub-chunks per outer chunk
    int B;           // block size
    int k;           // top-k
    int n_sink, n_local;
    int64_t M;       // sub-chunks
    int64_t nb;      // blocks
    int D;           // H_q * d_h
    int fp_groups;   // 256-dimension column groups of the fingerprint reduction
    float theta, sigma, attn_scale;
};

// Workspace regions (byte offsets from the workspace base).
struct WsLayout {
    size_t status;      // int32 status word (+ padding)
    size_t fp_ss;       // fp32 [M][fp_groups]: sums of squares of the fingerprint's column groups
    size_t gram;        // fp32 [M][S_max]   cosine of sub-chunk i with i+d
    size_t anchor;      // int32 [M]         1 if sub-chunk i opens a cluster
    size_t logits;      // fp32 [M][H_q][nb]     (block size > 1 only)
    size_t tok_split;   // bf16 [3][H_kv][M][g][128]  fingerprint parts (block size 1 only)
    size_t tok_part;    // float2 [M][H_q][ranges]    per-range softmax partials (block size 1 only)
    size_t tok_list;    // int32 [M][slots]           distant token list of each unit (block size 1 only)
    size_t tok_pack_k;  // bf16 [M][H_kv][slots][128] distant keys of each unit, packed (block size 1 only)
    size_t tok_pack_v;  // bf16 [M][H_kv][slots][128] distant values, packed
    size_t tok_count;   // int32 [M]                  distant keys of each unit
    size_t topk_hist;   // int32 [M][kTopkPasses][256] multi-CTA top-k scratch (block size 1 only)
    size_t topk_state;  // int32 [M][kTopkPasses + 1][4]
    size_t topk_counts; // int2 [M][topk chunks]
    size_t stats;       // fp32 [M][H_q][2]  (row max, 1 / row sum)
    size_t scores;      // fp32 [M][nb]
    size_t total;
};

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int derive(const scale_params_t* p, Derived* d);
WsLayout ws_layout(const Derived& d);

// Unit table as the kernels see it.
struct Units {
    const int32_t* unit_start;  // SCR only
    const int32_t* n_units;     // SCR only (device)
    int per_subchunk;
    int64_t N;
    int L;
    int M;
};

// Units starting in [tok_begin, tok_end): [first, first + count) with count
// bounded by max_units; both modes.
__device__ __forceinline__ int units_total(const Units& t)
{
    return t.per_subchunk ? t.M : *t.n_units;
}

// First unit whose first sub-chunk index is >= sc (binary search in SCR mode).
__device__ __forceinline__ int unit_lower_bound(const Units& t, int sc)
{
    if (t.per_subchunk) return sc < t.M ? sc : t.M;
    int lo = 0, hi = *t.n_units;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (t.unit_start[mid] < sc) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

// The unit that contains sub-chunk sc (units tile the sub-chunks in order).
__device__ __forceinline__ int unit_of_subchunk(const Units& t, int sc)
{
    return unit_lower_bound(t, sc + 1) - 1;
}

__device__ __forceinline__ void unit_range(const Units& t, int u, int* anchor, int64_t* s,
                                           int64_t* e)
{
    int a, b;
    if (t.per_subchunk) {
        a = u;
        b = u + 1;
    } else {
        a = t.unit_start[u];
        b = t.unit_start[u + 1];
    }
    *anchor = a;
    *s = static_cast<int64_t>(a) * t.L;
    const int64_t ee = static_cast<int64_t>(b) * t.L;
    *e = ee < t.N ? ee : t.N;
}

// Where token t's K and V rows live: row t of contiguous [N][H_kv][128]
// tensors (page_table == nullptr), or row page_table[t / page_size] *
// page_size + t % page_size of a page pool [num_pages * page_size][H_kv][128].
struct KvPaging {
    const int32_t* page_table;
    int page_size;
    int64_t num_pages;
    int64_t N;
    int64_t pool_rows;  // rows of the pool (N when contiguous)
};

// Row of token t, or -1 for t >= N or a page-table entry outside the pool.
__device__ __forceinline__ int64_t kv_row(const KvPaging& pg, int64_t t)
{
    if (t >= pg.N) return -1;
    if (!pg.page_table) return t;
    const int64_t lp = t / pg.page_size;
    const int64_t page = pg.page_table[lp];
    if (page < 0 || page >= pg.num_pages) return -1;
    return page * pg.page_size + (t - lp * pg.page_size);
}

// TMA coordinate of token t's row: rows that do not exist map past the end of
// the tensor, where TMA fills zeros.
__device__ __forceinline__ int32_t kv_row_tma(const KvPaging& pg, int64_t t)
{
    const int64_t r = kv_row(pg, t);
    return static_cast<int32_t>(r < 0 ? pg.pool_rows : r);
}

__device__ __forceinline__ void record_status(int32_t* status, int32_t code)
{
    atomicCAS(status, 0, code);
}

// ---- launchers (defined in the .cu files) ----
cudaError_t launch_build_reps(const Derived& d, const void* q, const void* k, const KvPaging& pg,
                              float* reps, float* fingerprints, int32_t* unit_start, int32_t* n_units,
                              uint8_t* ws, cudaStream_t st);
// Step (a) over the outer chunks [c_begin, c_end), appending their units to
// unit_start after the *n_units units of the chunks before c_begin.
cudaError_t launch_build_reps_range(const Derived& d, const void* q, const void* k, const KvPaging& pg,
                                    float* reps, float* fingerprints, int32_t* unit_start,
                                    int32_t* n_units, int c_begin, int c_end, uint8_t* ws,
                                    cudaStream_t st);
int outer_chunks(const Derived& d);
cudaError_t launch_select(const Derived& d, int mode, int64_t tok_begin, int64_t tok_end,
                          const float* reps, const float* fingerprints, const int32_t* unit_start,
                          const int32_t* n_units, int32_t* sel_blocks, int32_t* sel_count,
                          float* sel_scores, uint8_t* ws, uint64_t timeout_ns, cudaStream_t st);
cudaError_t launch_sparse_prefill(const Derived& d, int mode, int64_t tok_begin, int64_t tok_end,
                                  const void* q, const void* k, const void* v, const KvPaging& pg,
                                  const int32_t* unit_start, const int32_t* n_units,
                                  const int32_t* sel_blocks, const int32_t* sel_count, void* out,
                                  uint8_t* ws, uint64_t timeout_ns, cudaStream_t st);
cudaError_t launch_wait_selftest(uint8_t* ws, uint64_t timeout_ns, cudaStream_t st);
// Scratch of the multi-CTA top-k (units with more than 64K candidates).
// Radix passes of the multi-CTA top-k (8-bit digits of a 32-bit key).
constexpr int kTopkPasses = 4;
struct TopkScratch {
    int32_t* hist;    // [units][kTopkPasses][256]
    int32_t* state;   // [units][kTopkPasses + 1][4]
    int2* counts;     // [units][max_chunks]
    int max_chunks;   // topk_max_chunks(d)
};
int topk_max_chunks(const Derived& d);
cudaError_t launch_topk(const Derived& d, const Units& ut, int sc_begin, int sc_end, const float* scores,
                        int32_t* sel, int32_t* sel_count, cudaStream_t st, const int32_t* gate = nullptr,
                        const TopkScratch* scratch = nullptr);
cudaError_t launch_select_tokens(const Derived& d, int mode, int64_t tok_begin, int64_t tok_end,
                                 const void* k, const KvPaging& pg, const float* fingerprints,
                                 const int32_t* unit_start,
                                 const int32_t* n_units, int32_t* sel, int32_t* sel_count,
                                 float* sel_scores, uint8_t* ws, uint64_t timeout_ns, cudaStream_t st);
// Tokens per CTA of the token-level scoring kernels.
int tok_range(const Derived& d);
// Decode step (decode.cu).
size_t decode_cache_bytes(const Derived& d);
size_t decode_ws_bytes(const Derived& d, int splits);
int decode_splits();
cudaError_t launch_decode_step(const Derived& d, int64_t t, const void* q, const void* k, const void* v,
                               uint8_t* cache, void* out, uint8_t* ws, uint64_t timeout_ns, cudaStream_t st);

// Packed distant rows per (unit, KV head) at block size 1: n_sink + k rounded
// up to a multiple of 128.
int tok_slots(const Derived& d);

// Distant segments per unit the attention kernel may meet for these parameters.
int64_t max_distant_segments(const Derived& d);

}  // namespace scale
