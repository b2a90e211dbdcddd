// select.cu -- steps (b) and (c) of the SCR prefill path: cluster-level
// retrieval with head soft-voting (Eq. 9, Sec. V-A3 "Selection function
// instantiation") over block representative keys, then a deterministic top-k.
//
//   k_logits  z[u][h][b] = sigma * v_a(u)^(h) . r_b^(h/g)   (tcgen05 MMA per KV head:
//             128 (unit, head) rows x 128 blocks; both fp32 operands split
//             into three bf16 parts, six part products accumulated in fp32)
//   k_stats   per (u, h): max_b z and 1 / sum_b exp(z - max) over the candidates
//   k_vote    score[u][b] = sum_h exp(z[u][h][b] - max) / sum   (heads in order)
//   k_topk    up to 4096 candidates a bitonic sort of (score, -b) keys in
//             shared memory, beyond that a radix select of the k-th largest
//             key and an index-ordered compaction (and, with a scratch area
//             and more than 64K candidates, the multi-CTA form below): output
//             ascending, ties to the lower b.
//
// Candidates of unit u are the blocks with a token in [n_sink, W_u),
// W_u = max(0, s_u - n_local): the contiguous range [b_lo, b_hi(u)).
#include <cuda_bf16.h>

#include <cmath>

#include "ptx_sm103.cuh"
#include "scale_internal.h"

namespace scale {
namespace {

struct SelArgs {
    Units ut;
    int sc_begin, sc_end;  // sub-chunk range of units to process
    int Hq, g;
    int64_t nb;
    int B, k, n_sink, n_local;
    float sigma;
    const int32_t* gate;  // nullable: the top-k runs only when *gate != 0
    int32_t* status;      // device status word (bounded waits of k_logits)
    uint64_t timeout_ns;
};

__device__ __forceinline__ void cand_range(const SelArgs& a, int64_t s, int64_t* lo, int64_t* hi)
{
    const int64_t W = s - a.n_local > 0 ? s - a.n_local : 0;
    *lo = a.n_sink / a.B;                 // first block with (b+1)B > n_sink
    *hi = (W + a.B - 1) / a.B;            // one past the last block with bB < W
    if (*hi > a.nb) *hi = a.nb;
    if (*hi < *lo) *hi = *lo;
}

// Tensor-core logits. Grid: (unit tiles of 128 / g units, 128-block tiles,
// KV heads j). Rows of the A operand are the (unit, query head of KV head j)
// pairs of the tile (row ul * g + hl: head j g + hl of unit u0 + ul, the
// anchor's fingerprint slice), columns of B are the representatives of blocks
// [b0, b0 + 128) of KV head j. Both are fp32; every value x is split into
// three bf16 parts x1 + x2 + x3 = x exactly (x1 = bf16(x), x2 = bf16(x - x1),
// x3 = x - x1 - x2), written by the threads straight into the 128-byte-
// swizzled K-major layout of the MMA. The six part products a_i b_j with
// i + j <= 4 are exact in fp32 and are accumulated in fp32 in TMEM; the three
// dropped ones are below 2^-24 of |a| |b|. Only candidate blocks of each row's
// unit are written, as before.
constexpr int kLtThreads = 256;
constexpr uint32_t kLtPart = 128 * 128 * 2;   // one bf16 part: 128 rows x 128 columns
constexpr uint32_t kLtHalf = kLtPart / 2;     // one 64-column half
constexpr uint32_t kLtSmem = 6 * kLtPart + 1024;
static_assert(kLtSmem <= 227 * 1024, "logits shared memory");

__device__ __forceinline__ void split_bf16x3(float x, __nv_bfloat16& p1, __nv_bfloat16& p2, __nv_bfloat16& p3)
{
    p1 = __float2bfloat16_rn(x);
    const float r1 = x - __bfloat162float(p1);
    p2 = __float2bfloat16_rn(r1);
    p3 = __float2bfloat16_rn(r1 - __bfloat162float(p2));
}

// Four consecutive fp32 values of row r, columns [c, c + 4), into the three
// bf16 parts at `base` (part s at base + s * kLtPart): 8 bytes per part, at
// the 128-byte-swizzled K-major position of (r, c).
__device__ __forceinline__ void put_split4(uint8_t* base, int r, int c, float4 v)
{
    __nv_bfloat16 p[3][4];
    split_bf16x3(v.x, p[0][0], p[1][0], p[2][0]);
    split_bf16x3(v.y, p[0][1], p[1][1], p[2][1]);
    split_bf16x3(v.z, p[0][2], p[1][2], p[2][2]);
    split_bf16x3(v.w, p[0][3], p[1][3], p[2][3]);
    const int hf = c >> 6, cc = c & 63;  // half, column in the half
    const uint32_t off = hf * kLtHalf + (r >> 3) * 1024 + (r & 7) * 128 + ((((cc >> 3) ^ (r & 7))) << 4) +
                         (cc & 7) * 2;
#pragma unroll
    for (int s = 0; s < 3; ++s) {
        uint2 w;
        w.x = static_cast<uint32_t>(__bfloat16_as_ushort(p[s][0])) |
              (static_cast<uint32_t>(__bfloat16_as_ushort(p[s][1])) << 16);
        w.y = static_cast<uint32_t>(__bfloat16_as_ushort(p[s][2])) |
              (static_cast<uint32_t>(__bfloat16_as_ushort(p[s][3])) << 16);
        *reinterpret_cast<uint2*>(base + s * kLtPart + off) = w;
    }
}

__global__ void __launch_bounds__(kLtThreads, 1) k_logits(SelArgs a, const float* __restrict__ fp,
                                                          const float* __restrict__ reps,
                                                          float* __restrict__ logits)
{
    using namespace scale_ptx;
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint64_t d_full;
    __shared__ uint32_t tmem_slot;
    __shared__ int64_t s_lo[128], s_hi[128];
    __shared__ int s_anchor[128];
    __shared__ int any;
    const int U = 128 / a.g;  // units per tile
    const int u_first = unit_lower_bound(a.ut, a.sc_begin);
    const int u_end = unit_lower_bound(a.ut, a.sc_end);
    const int u0 = u_first + static_cast<int>(blockIdx.x) * U;
    if (u0 >= u_end) return;
    const int n_u = (u_end - u0 < U) ? u_end - u0 : U;
    const int rows = n_u * a.g;
    const int j = blockIdx.z;
    const int64_t b0 = static_cast<int64_t>(blockIdx.y) * 128;
    const int D = a.Hq * kHeadDim;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    // The tile is needed only if some unit's candidate range meets [b0, b0 + 128).
    if (tid == 0) any = 0;
    __syncthreads();
    if (tid < n_u) {
        int64_t s, e, lo, hi;
        int anc;
        unit_range(a.ut, u0 + tid, &anc, &s, &e);
        cand_range(a, s, &lo, &hi);
        s_lo[tid] = lo;
        s_hi[tid] = hi;
        s_anchor[tid] = anc;
        if (lo < hi && lo < b0 + 128 && hi > b0) atomicOr(&any, 1);
    }
    __syncthreads();
    if (!any) return;

    uint8_t* smem = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
    uint8_t* abuf = smem;                // A parts 0..2
    uint8_t* bbuf = smem + 3 * kLtPart;  // B parts 0..2
    // 128 rows x 32 float4 per operand; a warp reads one 512-byte row
    for (int x = tid; x < 128 * 32; x += kLtThreads) {
        const int r = x >> 5, c = (x & 31) * 4;
        float4 va = make_float4(0.f, 0.f, 0.f, 0.f), vb = va;
        if (r < rows) {
            const int ul = r / a.g, hl = r % a.g;
            va = *reinterpret_cast<const float4*>(fp + static_cast<int64_t>(s_anchor[ul]) * D +
                                                  (j * a.g + hl) * kHeadDim + c);
        }
        if (b0 + r < a.nb) vb = *reinterpret_cast<const float4*>(reps + (j * a.nb + b0 + r) * kHeadDim + c);
        put_split4(abuf, r, c, va);
        put_split4(bbuf, r, c, vb);
    }
    fence_proxy_async_smem();
    if (tid == 0) {
        mbar_init(&d_full, 1);
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc(&tmem_slot, 128);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (tid == 0) {
        const uint32_t idesc = idesc_bf16_f32(128, 128, 0);
        const uint64_t ad = sdesc_sw128(smem_addr(abuf), 16, 1024);
        const uint64_t bd = sdesc_sw128(smem_addr(bbuf), 16, 1024);
        constexpr uint64_t kPartStep = kLtPart >> 4;
        // (A part, B part): the products a_i b_j with i + j <= 4 (parts from 1)
        constexpr int kPa[6] = {0, 0, 1, 0, 1, 2};
        constexpr int kPb[6] = {0, 1, 0, 2, 1, 0};
#pragma unroll
        for (int i = 0; i < 6; ++i)
            mma_ss_k128<kLtHalf>(tmem, ad + kPa[i] * kPartStep, bd + kPb[i] * kPartStep, idesc, i > 0 ? 1u : 0u);
        mma_commit(&d_full);
    }
    bool done = true;
    if (warp < 4) {
        // epilogue: thread = row (TMEM lane) warp * 32 + lane
        done = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(&d_full, 0, a.timeout_ns, nullptr));
        if (done) {
            tc_fence_after();
            const uint32_t lane_base = tmem + (static_cast<uint32_t>(warp * 32) << 16);
            uint32_t zr[128];
#pragma unroll
            for (int cc = 0; cc < 4; ++cc)
                tmem_ld32(lane_base + cc * 32, *reinterpret_cast<uint32_t(*)[32]>(&zr[cc * 32]));
            tmem_ld_wait();
            const int r = warp * 32 + lane;
            if (r < rows) {
                const int ul = r / a.g, hl = r % a.g;
                const int64_t lo = s_lo[ul] > b0 ? s_lo[ul] : b0;
                const int64_t hi = s_hi[ul] < b0 + 128 ? s_hi[ul] : b0 + 128;
                float* dst = logits + (static_cast<int64_t>(u0 + ul) * a.Hq + j * a.g + hl) * a.nb + b0;
                const int c_lo = static_cast<int>(lo - b0), c_hi = static_cast<int>(hi - b0);
#pragma unroll
                for (int c = 0; c < 128; ++c)
                    if (c >= c_lo && c < c_hi) dst[c] = a.sigma * __uint_as_float(zr[c]);
            }
        } else if (lane == 0) {
            record_status(a.status, SCALE_ERR_TIMEOUT);
        }
    } else if (warp == 4 && lane == 0) {
        // TMEM is freed only after the MMAs completed (bounded)
        mbar_wait_bounded(&d_full, 0, a.timeout_ns, nullptr);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 128);
    }
}

// One warp per (unit, head): row max and 1 / sum of exp(z - max) over the candidates.
__global__ void __launch_bounds__(256) k_stats(SelArgs a, const float* __restrict__ logits,
                                               float* __restrict__ stats)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int u_first = unit_lower_bound(a.ut, a.sc_begin);
    const int u_end = unit_lower_bound(a.ut, a.sc_end);
    const int64_t uh = static_cast<int64_t>(blockIdx.x) * 8 + warp;
    const int u = u_first + static_cast<int>(uh / a.Hq);
    const int h = static_cast<int>(uh % a.Hq);
    if (u >= u_end) return;
    int anc;
    int64_t s, e, lo, hi;
    unit_range(a.ut, u, &anc, &s, &e);
    cand_range(a, s, &lo, &hi);
    if (lo >= hi) return;
    const float* z = logits + (static_cast<int64_t>(u) * a.Hq + h) * a.nb;
    // Eight loads in flight per lane; each lane still combines its values in
    // index order, so the result does not depend on the batching.
    constexpr int kIn = 8;
    float m = -INFINITY;
    for (int64_t b0 = lo + lane; b0 < hi; b0 += 32 * kIn) {
        float x[kIn];
#pragma unroll
        for (int i = 0; i < kIn; ++i) x[i] = b0 + 32 * i < hi ? z[b0 + 32 * i] : -INFINITY;
#pragma unroll
        for (int i = 0; i < kIn; ++i) m = fmaxf(m, x[i]);
    }
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    float sum = 0.f;
    for (int64_t b0 = lo + lane; b0 < hi; b0 += 32 * kIn) {
        float x[kIn];
#pragma unroll
        for (int i = 0; i < kIn; ++i) x[i] = b0 + 32 * i < hi ? z[b0 + 32 * i] : 0.f;
#pragma unroll
        for (int i = 0; i < kIn; ++i)
            if (b0 + 32 * i < hi) sum += expf(x[i] - m);
    }
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
    if (lane == 0) {
        stats[(static_cast<int64_t>(u) * a.Hq + h) * 2] = m;
        stats[(static_cast<int64_t>(u) * a.Hq + h) * 2 + 1] = 1.0f / sum;
    }
}

// score[u][b] = sum over heads (in order) of exp(z - max) / sum; NaN off the candidates.
__global__ void __launch_bounds__(256) k_vote(SelArgs a, const float* __restrict__ logits,
                                              const float* __restrict__ stats,
                                              float* __restrict__ scores)
{
    const int u_first = unit_lower_bound(a.ut, a.sc_begin);
    const int u_end = unit_lower_bound(a.ut, a.sc_end);
    const int u = u_first + blockIdx.y;
    if (u >= u_end) return;
    const int64_t b = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (b >= a.nb) return;
    int anc;
    int64_t s, e, lo, hi;
    unit_range(a.ut, u, &anc, &s, &e);
    cand_range(a, s, &lo, &hi);
    float score = __int_as_float(0x7FC00000);
    if (b >= lo && b < hi) {
        score = 0.f;
        const float* zb = logits + static_cast<int64_t>(u) * a.Hq * a.nb + b;
        const float* sb = stats + static_cast<int64_t>(u) * a.Hq * 2;
        // Eight heads' loads in flight at a time, added in head order.
        constexpr int kIn = 8;
        for (int h0 = 0; h0 < a.Hq; h0 += kIn) {
            float z[kIn], mx[kIn], inv[kIn];
#pragma unroll
            for (int i = 0; i < kIn; ++i) {
                const int h = h0 + i < a.Hq ? h0 + i : a.Hq - 1;
                z[i] = zb[static_cast<int64_t>(h) * a.nb];
                mx[i] = sb[2 * h];
                inv[i] = sb[2 * h + 1];
            }
#pragma unroll
            for (int i = 0; i < kIn; ++i)
                if (h0 + i < a.Hq) score += expf(z[i] - mx[i]) * inv[i];
        }
    }
    scores[static_cast<int64_t>(u) * a.nb + b] = score;
}

// Order-preserving map of a float onto uint32 (larger float -> larger key).
__device__ __forceinline__ uint32_t float_key(float f)
{
    const uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

constexpr int kTopkThreads = 1024;
constexpr int kSortMax = 4096;     // candidates up to which the top-k sorts instead

// The k picks among np (a power of two, at most kSortMax) 64-bit keys
// (~float_key(score), candidate index) in shared memory, written to out in
// ascending candidate order (candidate i is block lo + i): a bitonic sort puts
// the picks first (higher score first, equal scores by lower index), their
// indices are marked in a bitmap (bm: np / 32 + 1 words) and written in order
// after one scan. Called by all kTopkThreads threads of the CTA.
__device__ void topk_sort_emit(uint64_t* sk, uint32_t* bm, int np, int64_t lo, int k, int32_t* out)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int size = 2; size <= np; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = threadIdx.x; i < np; i += blockDim.x) {
                const int l = i ^ stride;
                if (l > i) {
                    const uint64_t x = sk[i], y = sk[l];
                    if ((x > y) == ((i & size) == 0)) {
                        sk[i] = y;
                        sk[l] = x;
                    }
                }
            }
            __syncthreads();
        }
    for (int w = threadIdx.x; w < np / 32 + 1; w += blockDim.x) bm[w] = 0u;
    __syncthreads();
    for (int r = threadIdx.x; r < k; r += blockDim.x) {
        const uint32_t i = static_cast<uint32_t>(sk[r]);
        atomicOr(&bm[i >> 5], 1u << (i & 31));
    }
    __syncthreads();
    // ascending output: word t of the bitmap to thread t, exclusive scan of the counts
    __shared__ int s_wsum[4];
    const int nwords = (np + 31) / 32;
    uint32_t word = threadIdx.x < nwords ? bm[threadIdx.x] : 0u;
    const int c = __popc(word);
    int inc = c;
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xFFFFFFFFu, inc, o);
        if (lane >= o) inc += y;
    }
    if (lane == 31 && warp < 4) s_wsum[warp] = inc;
    __syncthreads();
    if (threadIdx.x < nwords) {
        int p = inc - c;
        for (int w = 0; w < warp; ++w) p += s_wsum[w];
        while (word) {
            const int bit = __ffs(word) - 1;
            word &= word - 1;
            out[p++] = static_cast<int32_t>(lo + 32 * threadIdx.x + bit);
        }
    }
}
constexpr int kTopkUnroll = 16;  // independent loads in flight per thread

// One CTA per unit. Up to kSortMax candidates, a bitonic sort in shared
// memory of the 64-bit keys (~float_key(score), index) puts the picks first
// (higher score first, equal scores by lower index); their indices are marked
// in a bitmap and written in ascending order after one scan. Beyond that, the
// k-th largest key T is found with four 8-bit radix passes (16 coalesced
// loads in flight per thread); the selected blocks are those with key > T
// plus the lowest-indexed ones with key == T, emitted in ascending block
// order: every warp owns a contiguous segment, counts its picks, and after
// one scan over the warps writes them in order with warp-level prefix sums.
// Both give the same selection.
__global__ void __launch_bounds__(kTopkThreads) k_topk(SelArgs a, const float* __restrict__ scores,
                                                       int32_t* __restrict__ sel,
                                                       int32_t* __restrict__ sel_count)
{
    __shared__ int hist[256];
    __shared__ __align__(16) int whist[kTopkThreads / 32][256];  // per-warp histograms, or the sort keys
    static_assert(sizeof(whist) >= kSortMax * sizeof(uint64_t), "sort buffer");
    __shared__ uint32_t s_prefix;
    __shared__ int s_need;
    if (a.gate && !*a.gate) return;
    const int u_first = unit_lower_bound(a.ut, a.sc_begin);
    const int u_end = unit_lower_bound(a.ut, a.sc_end);
    const int u = u_first + blockIdx.x;
    if (u >= u_end) return;
    int anc;
    int64_t s, e, lo, hi;
    unit_range(a.ut, u, &anc, &s, &e);
    cand_range(a, s, &lo, &hi);
    const int64_t n = hi - lo;
    int32_t* out = sel + static_cast<int64_t>(u) * a.k;
    const float* sc = scores + static_cast<int64_t>(u) * a.nb;

    if (n <= a.k) {
        for (int i = threadIdx.x; i < a.k; i += blockDim.x) out[i] = (i < n) ? static_cast<int32_t>(lo + i) : -1;
        if (threadIdx.x == 0) sel_count[u] = static_cast<int32_t>(n);
        return;
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (n <= kSortMax) {
        uint64_t* sk = reinterpret_cast<uint64_t*>(&whist[0][0]);
        int np = 1;
        while (np < n) np <<= 1;
        for (int i = threadIdx.x; i < np; i += blockDim.x)
            sk[i] = i < n ? (static_cast<uint64_t>(~float_key(sc[lo + i])) << 32) | static_cast<uint32_t>(i)
                          : ~0ull;  // padding sorts last
        __syncthreads();
        topk_sort_emit(sk, reinterpret_cast<uint32_t*>(hist), np, lo, a.k, out);
        if (threadIdx.x == 0) sel_count[u] = a.k;  // n > k: exactly k picks
        return;
    }
    if (threadIdx.x == 0) {
        s_prefix = 0;
        s_need = a.k;
    }
    uint32_t mask = 0;
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int i = threadIdx.x; i < (kTopkThreads / 32) * 256; i += blockDim.x) (&whist[0][0])[i] = 0;
        __syncthreads();
        const uint32_t prefix = s_prefix;
        // Every warp counts into its own histogram (keys of similar magnitude
        // share digits, so one shared histogram would serialise on a few bins).
        for (int64_t b0 = lo; b0 < hi; b0 += kTopkUnroll * static_cast<int64_t>(blockDim.x)) {
            uint32_t key[kTopkUnroll];
#pragma unroll
            for (int j = 0; j < kTopkUnroll; ++j) {
                const int64_t b = b0 + j * blockDim.x + threadIdx.x;
                key[j] = b < hi ? float_key(sc[b]) : 0u;
            }
#pragma unroll
            for (int j = 0; j < kTopkUnroll; ++j) {
                const int64_t b = b0 + j * blockDim.x + threadIdx.x;
                const bool in = b < hi && (key[j] & mask) == prefix;
                if (in) atomicAdd(&whist[warp][(key[j] >> shift) & 255u], 1);
            }
        }
        __syncthreads();
        for (int i = threadIdx.x; i < 256; i += blockDim.x) {
            int c = 0;
            for (int w = 0; w < kTopkThreads / 32; ++w) c += whist[w][i];
            hist[i] = c;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            int need = s_need, cum = 0, d = 255;
            for (; d > 0; --d) {
                if (cum + hist[d] >= need) break;
                cum += hist[d];
            }
            s_need = need - cum;
            s_prefix = prefix | (static_cast<uint32_t>(d) << shift);
        }
        mask |= 255u << shift;
        __syncthreads();
    }
    const uint32_t T = s_prefix;
    const int need_eq = s_need;  // how many keys equal to T to take, lowest b first
    // Ordered compaction: warp w owns the contiguous segment [w0, w1); lane l
    // reads keys w0 + 128 i + 4 l .. + 3, so every step is one coalesced 512-byte
    // read and index order within the warp is (step, lane, j).
    const int nw = blockDim.x >> 5;
    const int64_t seg = ((n + nw - 1) / nw + 127) / 128 * 128;
    const int64_t w0 = lo + seg * warp;
    const int64_t w1 = (w0 + seg < hi) ? w0 + seg : hi;
    auto load4 = [&](int64_t b, uint32_t (&key)[4]) {
#pragma unroll
        for (int j = 0; j < 4; ++j) key[j] = (b + j < w1) ? float_key(sc[b + j]) : 0u;
    };
    int n_gt = 0, n_eq = 0;
    for (int64_t b = w0 + 4 * lane; b < w1; b += 128) {
        uint32_t key[4];
        load4(b, key);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            n_gt += (b + j < w1) && key[j] > T;
            n_eq += (b + j < w1) && key[j] == T;
        }
    }
    for (int o = 16; o > 0; o >>= 1) {
        n_gt += __shfl_xor_sync(0xFFFFFFFFu, n_gt, o);
        n_eq += __shfl_xor_sync(0xFFFFFFFFu, n_eq, o);
    }
    __shared__ int s_take[kTopkThreads / 32], s_pos[kTopkThreads / 32], s_taken;
    if (lane == 0) {
        s_take[warp] = n_eq;  // equal keys of this warp, for now
        s_pos[warp] = n_gt;   // keys above T of this warp, for now
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int eq_before = 0, pos = 0;
        for (int w = 0; w < nw; ++w) {
            const int e = s_take[w], g = s_pos[w];
            int take = need_eq - eq_before;
            take = take < 0 ? 0 : (take > e ? e : take);
            eq_before += e;
            s_take[w] = take;
            s_pos[w] = pos;
            pos += g + take;
        }
        s_taken = pos;
    }
    __syncthreads();
    const int taken = s_taken;
    int pos = s_pos[warp], take_eq = s_take[warp];
    for (int64_t b = w0 + 4 * lane; b < w1; b += 128) {
        uint32_t key[4];
        load4(b, key);
        int gt_l = 0, eq_l = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            gt_l += (b + j < w1) && key[j] > T;
            eq_l += (b + j < w1) && key[j] == T;
        }
        // exclusive prefix over lanes of the equal keys
        int eq_inc = eq_l;
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, eq_inc, o);
            if (lane >= o) eq_inc += y;
        }
        const int eq_tot = __shfl_sync(0xFFFFFFFFu, eq_inc, 31);
        int eq_rank = eq_inc - eq_l;  // equal keys before this lane in this step
        // picks of this lane: keys above T and the equal keys still to take
        int pk[4], n_pk = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            pk[j] = 0;
            if (b + j < w1) {
                if (key[j] > T) pk[j] = 1;
                else if (key[j] == T) pk[j] = (eq_rank++ < take_eq);
            }
            n_pk += pk[j];
        }
        int pk_inc = n_pk;
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, pk_inc, o);
            if (lane >= o) pk_inc += y;
        }
        int p = pos + pk_inc - n_pk;
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (pk[j]) out[p++] = static_cast<int32_t>(b + j);
        pos += __shfl_sync(0xFFFFFFFFu, pk_inc, 31);
        take_eq -= (eq_tot < take_eq ? eq_tot : take_eq);
    }
    for (int i = taken + threadIdx.x; i < a.k; i += blockDim.x) out[i] = -1;
    if (threadIdx.x == 0) sel_count[u] = taken;
}

// Steps (b)-(c) after the logits for units of at most kSortMax candidates,
// one CTA of kTopkThreads per unit: the per-head max and 1 / sum of k_stats,
// the soft vote of k_vote (scores written for every block, NaN off the
// candidates) and the sort path of k_topk, with the same arithmetic in the
// same order, so scores and selection equal those of the three kernels.
constexpr int kFusedMaxHeads = 256;
__global__ void __launch_bounds__(kTopkThreads) k_select_fused(SelArgs a, const float* __restrict__ logits,
                                                               float* __restrict__ scores,
                                                               int32_t* __restrict__ sel,
                                                               int32_t* __restrict__ sel_count)
{
    __shared__ float s_m[kFusedMaxHeads], s_inv[kFusedMaxHeads];
    __shared__ __align__(16) uint64_t sk[kSortMax];
    __shared__ uint32_t bm[kSortMax / 32 + 1];
    const int u_first = unit_lower_bound(a.ut, a.sc_begin);
    const int u_end = unit_lower_bound(a.ut, a.sc_end);
    const int u = u_first + blockIdx.x;
    if (u >= u_end) return;
    int anc;
    int64_t s, e, lo, hi;
    unit_range(a.ut, u, &anc, &s, &e);
    cand_range(a, s, &lo, &hi);
    const int64_t n = hi - lo;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int kIn = 8;
    // per-head statistics over the candidates (k_stats): one warp per head
    if (n > 0)
        for (int h = warp; h < a.Hq; h += kTopkThreads / 32) {
            const float* z = logits + (static_cast<int64_t>(u) * a.Hq + h) * a.nb;
            float m = -INFINITY;
            for (int64_t b0 = lo + lane; b0 < hi; b0 += 32 * kIn) {
                float x[kIn];
#pragma unroll
                for (int i = 0; i < kIn; ++i) x[i] = b0 + 32 * i < hi ? z[b0 + 32 * i] : -INFINITY;
#pragma unroll
                for (int i = 0; i < kIn; ++i) m = fmaxf(m, x[i]);
            }
            for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
            float sum = 0.f;
            for (int64_t b0 = lo + lane; b0 < hi; b0 += 32 * kIn) {
                float x[kIn];
#pragma unroll
                for (int i = 0; i < kIn; ++i) x[i] = b0 + 32 * i < hi ? z[b0 + 32 * i] : 0.f;
#pragma unroll
                for (int i = 0; i < kIn; ++i)
                    if (b0 + 32 * i < hi) sum += expf(x[i] - m);
            }
            for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
            if (lane == 0) {
                s_m[h] = m;
                s_inv[h] = 1.0f / sum;
            }
        }
    __syncthreads();
    // soft vote over the heads in order (k_vote); the candidates' sort keys
    int np = 1;
    while (np < n) np <<= 1;
    const bool sort = n > a.k;
    for (int64_t b = threadIdx.x; b < a.nb; b += kTopkThreads) {
        float score = __int_as_float(0x7FC00000);
        if (b >= lo && b < hi) {
            score = 0.f;
            const float* zb = logits + static_cast<int64_t>(u) * a.Hq * a.nb + b;
            for (int h0 = 0; h0 < a.Hq; h0 += kIn) {
                float z[kIn], mx[kIn], inv[kIn];
#pragma unroll
                for (int i = 0; i < kIn; ++i) {
                    const int h = h0 + i < a.Hq ? h0 + i : a.Hq - 1;
                    z[i] = zb[static_cast<int64_t>(h) * a.nb];
                    mx[i] = s_m[h];
                    inv[i] = s_inv[h];
                }
#pragma unroll
                for (int i = 0; i < kIn; ++i)
                    if (h0 + i < a.Hq) score += expf(z[i] - mx[i]) * inv[i];
            }
            if (sort)
                sk[b - lo] = (static_cast<uint64_t>(~float_key(score)) << 32) | static_cast<uint32_t>(b - lo);
        }
        scores[static_cast<int64_t>(u) * a.nb + b] = score;
    }
    int32_t* out = sel + static_cast<int64_t>(u) * a.k;
    if (!sort) {
        for (int i = threadIdx.x; i < a.k; i += blockDim.x) out[i] = (i < n) ? static_cast<int32_t>(lo + i) : -1;
        if (threadIdx.x == 0) sel_count[u] = static_cast<int32_t>(n);
        return;
    }
    for (int i = static_cast<int>(n) + threadIdx.x; i < np; i += kTopkThreads) sk[i] = ~0ull;  // padding sorts last
    __syncthreads();
    topk_sort_emit(sk, bm, np, lo, a.k, out);
    if (threadIdx.x == 0) sel_count[u] = a.k;  // n > k: exactly k picks
}

// ---- top-k over many candidates per unit: the same radix select and ordered
// output as k_topk, spread over CTAs of kChunk candidates (grid y = unit).

constexpr int kChunk = 2048;              // candidates per CTA and pass
constexpr int64_t kMultiCtaMin = 65536;   // more candidates than this: the multi-CTA form
constexpr int kChunkThreads = 256;

struct TopkState {
    uint32_t prefix;  // bits of the k-th key fixed so far
    int need;         // keys still to take at or below the prefix
    int done;         // 1: the unit's output is already complete
    int pad;
};
static_assert(sizeof(TopkState) == 4 * sizeof(int32_t), "TopkState is four int32 words");

__device__ __forceinline__ bool unit_cands(const SelArgs& a, int ui, int* u, int64_t* lo, int64_t* hi)
{
    const int u_first = unit_lower_bound(a.ut, a.sc_begin);
    const int u_end = unit_lower_bound(a.ut, a.sc_end);
    *u = u_first + ui;
    if (*u >= u_end) return false;
    int anc;
    int64_t s, e;
    unit_range(a.ut, *u, &anc, &s, &e);
    cand_range(a, s, lo, hi);
    return true;
}

// Per unit: small candidate sets are written out directly; otherwise the
// radix state starts (prefix 0, need k) and the four passes' histograms are
// cleared. state[u][i] is the state after the digits of i passes are fixed;
// the kernel that first needs state i + 1 derives it from state i and the
// histogram of pass i (its CTA 0 stores it for the kernels after it).
__global__ void __launch_bounds__(256) k_topk_init(SelArgs a, int32_t* __restrict__ sel,
                                                    int32_t* __restrict__ sel_count, int32_t* __restrict__ hist,
                                                    TopkState* __restrict__ state)
{
    if (a.gate && !*a.gate) return;
    int u;
    int64_t lo, hi;
    if (!unit_cands(a, blockIdx.x, &u, &lo, &hi)) return;
    const int64_t n = hi - lo;
    for (int i = threadIdx.x; i < kTopkPasses * 256; i += blockDim.x) hist[u * kTopkPasses * 256 + i] = 0;
    if (n <= a.k) {
        int32_t* out = sel + static_cast<int64_t>(u) * a.k;
        for (int i = threadIdx.x; i < a.k; i += blockDim.x) out[i] = (i < n) ? static_cast<int32_t>(lo + i) : -1;
        if (threadIdx.x == 0) {
            sel_count[u] = static_cast<int32_t>(n);
            state[u * (kTopkPasses + 1)] = TopkState{0u, 0, 1, 0};
        }
    } else if (threadIdx.x == 0) {
        state[u * (kTopkPasses + 1)] = TopkState{0u, a.k, 0, 0};
    }
}

// State after pass p (p >= 1): the digit of the k-th largest key at the
// shift of pass p - 1, from that pass's histogram and the state before it
// (the largest digit d whose keys, with those above it, reach `need`).
// Every thread of the CTA returns it; CTA 0 stores it.
__device__ TopkState topk_state_after(const int32_t* __restrict__ hist_u, TopkState* __restrict__ state_u,
                                      int p, bool store)
{
    __shared__ int h[256];
    __shared__ TopkState s_st;
    for (int i = threadIdx.x; i < 256; i += blockDim.x) h[i] = hist_u[(p - 1) * 256 + i];
    __syncthreads();
    if (threadIdx.x == 0) {
        TopkState stt = state_u[p - 1];
        int need = stt.need, cum = 0, d = 255;
        for (; d > 0; --d) {
            if (cum + h[d] >= need) break;
            cum += h[d];
        }
        stt.need = need - cum;
        stt.prefix |= static_cast<uint32_t>(d) << (24 - 8 * (p - 1));
        s_st = stt;
        if (store) state_u[p] = stt;
    }
    __syncthreads();
    return s_st;
}

// Radix pass p (shift 24 - 8 p): per-warp histograms of the digit at `shift`
// of the keys that match the prefix fixed by the passes before, added into
// the unit's histogram of pass p.
__global__ void __launch_bounds__(kChunkThreads) k_topk_hist(SelArgs a, const float* __restrict__ scores,
                                                             int32_t* __restrict__ hist,
                                                             TopkState* __restrict__ state, int p)
{
    __shared__ int wh[kChunkThreads / 32][256];
    if (a.gate && !*a.gate) return;
    int u;
    int64_t lo, hi;
    if (!unit_cands(a, blockIdx.y, &u, &lo, &hi)) return;
    TopkState* su = state + u * (kTopkPasses + 1);
    int32_t* hu = hist + u * kTopkPasses * 256;
    if (su[0].done) return;
    const int64_t c0 = lo + static_cast<int64_t>(blockIdx.x) * kChunk;
    if (c0 >= hi) return;
    const int shift = 24 - 8 * p;
    const TopkState stt = p == 0 ? su[0] : topk_state_after(hu, su, p, blockIdx.x == 0);
    const int64_t c1 = (c0 + kChunk < hi) ? c0 + kChunk : hi;
    const int warp = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < (kChunkThreads / 32) * 256; i += blockDim.x) (&wh[0][0])[i] = 0;
    __syncthreads();
    const uint32_t mask = shift == 24 ? 0u : (0xFFFFFFFFu << (shift + 8));
    const float* sc = scores + static_cast<int64_t>(u) * a.nb;
    constexpr int kPer = kChunk / kChunkThreads;
    uint32_t key[kPer];
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
        const int64_t b = c0 + j * kChunkThreads + threadIdx.x;
        key[j] = b < c1 ? float_key(sc[b]) : 0u;
    }
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
        const int64_t b = c0 + j * kChunkThreads + threadIdx.x;
        if (b < c1 && (key[j] & mask) == stt.prefix) atomicAdd(&wh[warp][(key[j] >> shift) & 255u], 1);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 256; i += blockDim.x) {
        int c = 0;
        for (int w = 0; w < kChunkThreads / 32; ++w) c += wh[w][i];
        if (c) atomicAdd(&hu[p * 256 + i], c);
    }
}

// Counts per chunk of the keys above the k-th key T and of the keys equal to it.
// The k-th key T is the prefix after the last pass (derived here, stored by CTA 0).
__global__ void __launch_bounds__(kChunkThreads) k_topk_count(SelArgs a, const float* __restrict__ scores,
                                                              const int32_t* __restrict__ hist,
                                                              TopkState* __restrict__ state,
                                                              int2* __restrict__ counts, int max_chunks)
{
    if (a.gate && !*a.gate) return;
    int u;
    int64_t lo, hi;
    if (!unit_cands(a, blockIdx.y, &u, &lo, &hi)) return;
    TopkState* su = state + u * (kTopkPasses + 1);
    if (su[0].done) return;
    const int64_t c0 = lo + static_cast<int64_t>(blockIdx.x) * kChunk;
    if (c0 >= hi) return;
    const TopkState stt = topk_state_after(hist + u * kTopkPasses * 256, su, kTopkPasses, blockIdx.x == 0);
    const int64_t c1 = (c0 + kChunk < hi) ? c0 + kChunk : hi;
    const float* sc = scores + static_cast<int64_t>(u) * a.nb;
    int gt = 0, eq = 0;
    for (int64_t b = c0 + threadIdx.x; b < c1; b += blockDim.x) {
        const uint32_t key = float_key(sc[b]);
        gt += key > stt.prefix;
        eq += key == stt.prefix;
    }
    for (int o = 16; o > 0; o >>= 1) {
        gt += __shfl_xor_sync(0xFFFFFFFFu, gt, o);
        eq += __shfl_xor_sync(0xFFFFFFFFu, eq, o);
    }
    __shared__ int sg[kChunkThreads / 32], se[kChunkThreads / 32];
    if ((threadIdx.x & 31) == 0) {
        sg[threadIdx.x >> 5] = gt;
        se[threadIdx.x >> 5] = eq;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int g = 0, e = 0;
        for (int w = 0; w < kChunkThreads / 32; ++w) {
            g += sg[w];
            e += se[w];
        }
        counts[static_cast<int64_t>(u) * max_chunks + blockIdx.x] = make_int2(g, e);
    }
}

// Per unit: output position and number of equal keys to take of every chunk
// (the equal keys are taken lowest index first); the -1 padding and the count.
__global__ void __launch_bounds__(32) k_topk_scan(SelArgs a, const TopkState* __restrict__ state,
                                                   int2* __restrict__ counts, int max_chunks,
                                                   int32_t* __restrict__ sel, int32_t* __restrict__ sel_count)
{
    if (a.gate && !*a.gate) return;
    int u;
    int64_t lo, hi;
    if (!unit_cands(a, blockIdx.x, &u, &lo, &hi)) return;
    if (state[u * (kTopkPasses + 1)].done) return;
    const TopkState stt = state[u * (kTopkPasses + 1) + kTopkPasses];
    const int n_chunks = static_cast<int>((hi - lo + kChunk - 1) / kChunk);
    int2* cu = counts + static_cast<int64_t>(u) * max_chunks;
    // Two prefix sums over the chunks, 32 at a time with the totals carried:
    // the equal keys before each chunk (how many of its equal keys it takes
    // follows), then the picks before it (its output position).
    const int lane = threadIdx.x;
    int eq_run = 0, pos_run = 0;
    for (int c0 = 0; c0 < n_chunks; c0 += 32) {
        const int c = c0 + lane;
        const int2 ge = c < n_chunks ? cu[c] : make_int2(0, 0);
        int eq_inc = ge.y;
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, eq_inc, o);
            if (lane >= o) eq_inc += y;
        }
        const int eq_before = eq_run + eq_inc - ge.y;
        int take = stt.need - eq_before;
        take = take < 0 ? 0 : (take > ge.y ? ge.y : take);
        const int picks = ge.x + take;
        int pos_inc = picks;
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, pos_inc, o);
            if (lane >= o) pos_inc += y;
        }
        if (c < n_chunks) cu[c] = make_int2(pos_run + pos_inc - picks, take);
        eq_run += __shfl_sync(0xFFFFFFFFu, eq_inc, 31);
        pos_run += __shfl_sync(0xFFFFFFFFu, pos_inc, 31);
    }
    if (lane == 0) sel_count[u] = pos_run;
    int32_t* out = sel + static_cast<int64_t>(u) * a.k;
    for (int i = pos_run + lane; i < a.k; i += 32) out[i] = -1;
}

// Ordered output of one chunk: every warp owns a contiguous segment (lane l
// reads 4 consecutive keys per step), counts its picks, and after a scan over
// the warps writes them in index order with warp prefix sums.
__global__ void __launch_bounds__(kChunkThreads) k_topk_emit(SelArgs a, const float* __restrict__ scores,
                                                             const TopkState* __restrict__ state,
                                                             const int2* __restrict__ counts, int max_chunks,
                                                             int32_t* __restrict__ sel)
{
    if (a.gate && !*a.gate) return;
    int u;
    int64_t lo, hi;
    if (!unit_cands(a, blockIdx.y, &u, &lo, &hi)) return;
    if (state[u * (kTopkPasses + 1)].done) return;
    const TopkState stt = state[u * (kTopkPasses + 1) + kTopkPasses];
    const int64_t c0 = lo + static_cast<int64_t>(blockIdx.x) * kChunk;
    if (c0 >= hi) return;
    const int64_t c1 = (c0 + kChunk < hi) ? c0 + kChunk : hi;
    const int2 pt = counts[static_cast<int64_t>(u) * max_chunks + blockIdx.x];
    const uint32_t T = stt.prefix;
    const float* sc = scores + static_cast<int64_t>(u) * a.nb;
    int32_t* out = sel + static_cast<int64_t>(u) * a.k;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int nw = kChunkThreads / 32;
    const int64_t seg = kChunk / nw;
    const int64_t w0 = c0 + seg * warp;
    const int64_t w1 = (w0 + seg < c1) ? w0 + seg : c1;
    int n_gt = 0, n_eq = 0;
    for (int64_t b = w0 + 4 * lane; b < w1; b += 128)
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (b + j < w1) {
                const uint32_t key = float_key(sc[b + j]);
                n_gt += key > T;
                n_eq += key == T;
            }
    for (int o = 16; o > 0; o >>= 1) {
        n_gt += __shfl_xor_sync(0xFFFFFFFFu, n_gt, o);
        n_eq += __shfl_xor_sync(0xFFFFFFFFu, n_eq, o);
    }
    __shared__ int s_take[nw], s_pos[nw];
    if (lane == 0) {
        s_take[warp] = n_eq;
        s_pos[warp] = n_gt;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int eq_before = 0, pos = pt.x;
        for (int w = 0; w < nw; ++w) {
            const int e = s_take[w], g = s_pos[w];
            int take = pt.y - eq_before;
            take = take < 0 ? 0 : (take > e ? e : take);
            eq_before += e;
            s_take[w] = take;
            s_pos[w] = pos;
            pos += g + take;
        }
    }
    __syncthreads();
    int pos = s_pos[warp], take_eq = s_take[warp];
    for (int64_t b = w0 + 4 * lane; b < w1; b += 128) {
        uint32_t key[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) key[j] = (b + j < w1) ? float_key(sc[b + j]) : 0u;
        int eq_l = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) eq_l += (b + j < w1) && key[j] == T;
        int eq_inc = eq_l;
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, eq_inc, o);
            if (lane >= o) eq_inc += y;
        }
        const int eq_tot = __shfl_sync(0xFFFFFFFFu, eq_inc, 31);
        int eq_rank = eq_inc - eq_l;
        int pk[4], n_pk = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            pk[j] = 0;
            if (b + j < w1) {
                if (key[j] > T) pk[j] = 1;
                else if (key[j] == T) pk[j] = (eq_rank++ < take_eq);
            }
            n_pk += pk[j];
        }
        int pk_inc = n_pk;
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, pk_inc, o);
            if (lane >= o) pk_inc += y;
        }
        int p = pos + pk_inc - n_pk;
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (pk[j]) out[p++] = static_cast<int32_t>(b + j);
        pos += __shfl_sync(0xFFFFFFFFu, pk_inc, 31);
        take_eq -= (eq_tot < take_eq ? eq_tot : take_eq);
    }
}

}  // namespace

int topk_max_chunks(const Derived& d) { return static_cast<int>((d.nb + kChunk - 1) / kChunk); }

cudaError_t launch_select(const Derived& d, int mode, int64_t tok_begin, int64_t tok_end,
                          const float* reps, const float* fingerprints, const int32_t* unit_start,
                          const int32_t* n_units, int32_t* sel_blocks, int32_t* sel_count,
                          float* sel_scores, uint8_t* ws, uint64_t timeout_ns, cudaStream_t st)
{
    const WsLayout lay = ws_layout(d);
    float* logits = reinterpret_cast<float*>(ws + lay.logits);
    float* stats = reinterpret_cast<float*>(ws + lay.stats);
    float* scores = sel_scores ? sel_scores : reinterpret_cast<float*>(ws + lay.scores);

    SelArgs a{};
    a.ut = Units{unit_start, n_units, mode == SCALE_MODE_PER_SUBCHUNK, d.N, d.L, static_cast<int>(d.M)};
    a.sc_begin = static_cast<int>(tok_begin / d.L);
    a.sc_end = static_cast<int>((tok_end + d.L - 1) / d.L);
    a.Hq = d.Hq;
    a.g = d.g;
    a.nb = d.nb;
    a.B = d.B;
    a.k = d.k;
    a.n_sink = d.n_sink;
    a.n_local = d.n_local;
    a.sigma = d.sigma;
    a.status = reinterpret_cast<int32_t*>(ws + kStatusOffset);
    a.timeout_ns = timeout_ns;
    const int max_units = a.sc_end - a.sc_begin;  // units in range <= sub-chunks in range
    if (max_units <= 0) return cudaSuccess;

    const int upt = 128 / d.g;  // units per logits tile
    // set on every launch: the attribute belongs to the current device
    cudaError_t e = cudaFuncSetAttribute(k_logits, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kLtSmem));
    if (e != cudaSuccess) return e;
    dim3 gl((max_units + upt - 1) / upt, static_cast<unsigned>((d.nb + 127) / 128), d.Hkv);
    k_logits<<<gl, kLtThreads, kLtSmem, st>>>(a, fingerprints, reps, logits);
    if (d.nb <= kSortMax && d.Hq <= kFusedMaxHeads && d.k <= kSortMax) {
        // every unit's candidates fit the sort: statistics, vote and top-k in one kernel
        k_select_fused<<<max_units, kTopkThreads, 0, st>>>(a, logits, scores, sel_blocks, sel_count);
        return cudaGetLastError();
    }
    const int64_t rows = static_cast<int64_t>(max_units) * d.Hq;
    k_stats<<<static_cast<unsigned>((rows + 7) / 8), 256, 0, st>>>(a, logits, stats);
    k_vote<<<dim3(static_cast<unsigned>((d.nb + 255) / 256), max_units), 256, 0, st>>>(a, logits, stats, scores);
    k_topk<<<max_units, kTopkThreads, 0, st>>>(a, scores, sel_blocks, sel_count);
    return cudaGetLastError();
}

cudaError_t launch_topk(const Derived& d, const Units& ut, int sc_begin, int sc_end, const float* scores,
                        int32_t* sel, int32_t* sel_count, cudaStream_t st, const int32_t* gate,
                        const TopkScratch* scratch)
{
    SelArgs a{};
    a.gate = gate;
    a.ut = ut;
    a.sc_begin = sc_begin;
    a.sc_end = sc_end;
    a.Hq = d.Hq;
    a.g = d.g;
    a.nb = d.nb;
    a.B = d.B;
    a.k = d.k;
    a.n_sink = d.n_sink;
    a.n_local = d.n_local;
    a.sigma = d.sigma;
    const int max_units = sc_end - sc_begin;
    if (max_units <= 0) return cudaSuccess;
    if (!scratch || d.nb <= kMultiCtaMin) {
        k_topk<<<max_units, kTopkThreads, 0, st>>>(a, scores, sel, sel_count);
        return cudaGetLastError();
    }
    // many candidates per unit: chunks of kChunk keys over the whole GPU
    auto* state = reinterpret_cast<TopkState*>(scratch->state);
    const int mc = scratch->max_chunks;
    const dim3 grid(static_cast<unsigned>(mc), static_cast<unsigned>(max_units));
    k_topk_init<<<max_units, 256, 0, st>>>(a, sel, sel_count, scratch->hist, state);
    for (int p = 0; p < kTopkPasses; ++p)
        k_topk_hist<<<grid, kChunkThreads, 0, st>>>(a, scores, scratch->hist, state, p);
    k_topk_count<<<grid, kChunkThreads, 0, st>>>(a, scores, scratch->hist, state, scratch->counts, mc);
    k_topk_scan<<<max_units, 32, 0, st>>>(a, state, scratch->counts, mc, sel, sel_count);
    k_topk_emit<<<grid, kChunkThreads, 0, st>>>(a, scores, state, scratch->counts, mc, sel);
    return cudaGetLastError();
}

}  // namespace scale
