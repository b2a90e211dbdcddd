// decode.cu -- one decode step with a selection cache.
//
// The paper's method targets prefill and leaves decode to the underlying
// engine, whose selection cache reuses a token selection across consecutive,
// highly similar decode queries (Sec. VII, TPOT). This file implements that
// step with the paper's own rules at C = 1 (Def. 1: a decode step processes
// one token):
//  - selection (Eq. 9 at block size 1): the query q_t of position t is the
//    unit's fingerprint; candidates n_sink <= c < W_t, W_t = max(0, t -
//    n_local); per-head softmax over the candidates, head soft-vote, top-k
//    tokens (ties to the lower index), ascending;
//  - cache (Eq. 8 / Algorithm 1 across steps): the query of the last step that
//    retrieved is the anchor; a step reuses the anchor's selection while
//    cos(q_t, anchor) >= theta and fewer than max_cluster_subchunks steps
//    have shared it, and retrieves (and becomes the anchor) otherwise;
//  - attention (Eq. 10 for one row): keys = sinks U selection U [W_t, t].
//
// Scoring one query against every key is a matrix-vector product: it runs on
// the CUDA cores, one warp per key, reading K once with 8-byte loads per lane
// (the step is bound by HBM, not by arithmetic). Whether the step retrieves is
// decided on the device, so a step never synchronises with the host.
#include <cuda_bf16.h>

#include <cmath>

#include "scale_internal.h"

namespace scale {
namespace {

// Decode cache layout (bytes from its base).
constexpr size_t kDecState = 0;     // int32[8]: valid, steps, retrieve, -, anchor position
constexpr size_t kDecUnits = 64;    // int32[2] unit table [t, t + 1] of the anchor, int32 n_units
constexpr size_t kDecAnchor = 256;  // fp32 [H_q * 128]
// selection int32 [k] and its count follow the anchor

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

struct DecArgs {
    int Hq, Hkv, g;
    int64_t t;          // position of the decode query (its K and V rows are present)
    int64_t cap;        // rows of K and V
    int n_sink, n_local, k, S_max;
    float theta, sigma, attn_scale_log2;
    int32_t* state;
    int32_t* units;     // [t_anchor, t_anchor + 1], then n_units
    float* anchor;
    int32_t* sel;
    int32_t* sel_count;
    float* z;           // [H_q][cap]
    float2* stats;      // [H_q] (max, 1 / sum)
    float* scores;      // [cap]
    float* part;        // [H_q][splits][130]: max, sum, o[128]
    int splits;
    float2* zpart;      // [chunks][H_q] (max, sum) of each candidate chunk
    int chunk;          // candidates per logits CTA
};

__host__ __device__ __forceinline__ int64_t window_start(const DecArgs& a, int64_t t)
{
    return t - a.n_local > 0 ? t - a.n_local : 0;
}

// Reuse decision and anchor update (one CTA of 256 threads).
__global__ void __launch_bounds__(256) k_dec_gate(DecArgs a, const __nv_bfloat16* __restrict__ q)
{
    __shared__ float red[3][8];
    const int D = a.Hq * kHeadDim;
    float dot = 0.f, nq = 0.f, na = 0.f;
    for (int i = threadIdx.x; i < D; i += blockDim.x) {
        const float x = __bfloat162float(q[i]);
        const float y = a.anchor[i];
        dot += x * y;
        nq += x * x;
        na += y * y;
    }
    for (int o = 16; o > 0; o >>= 1) {
        dot += __shfl_xor_sync(0xFFFFFFFFu, dot, o);
        nq += __shfl_xor_sync(0xFFFFFFFFu, nq, o);
        na += __shfl_xor_sync(0xFFFFFFFFu, na, o);
    }
    const int w = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) {
        red[0][w] = dot;
        red[1][w] = nq;
        red[2][w] = na;
    }
    __syncthreads();
    __shared__ int s_retrieve;
    if (threadIdx.x == 0) {
        float d = 0.f, a2 = 0.f, b2 = 0.f;
        for (int i = 0; i < 8; ++i) {
            d += red[0][i];
            a2 += red[1][i];
            b2 += red[2][i];
        }
        const float cs = (a2 > 0.f && b2 > 0.f) ? d / (sqrtf(a2) * sqrtf(b2)) : 0.f;  // zero norm: 0
        const int valid = a.state[0], steps = a.state[1];
        const bool reuse = valid && steps < a.S_max && cs >= a.theta;
        if (reuse) {
            a.state[1] = steps + 1;
            a.state[2] = 0;
        } else {
            a.state[0] = 1;
            a.state[1] = 1;
            a.state[2] = 1;
            a.state[4] = static_cast<int32_t>(a.t);
            a.units[0] = static_cast<int32_t>(a.t);
            a.units[1] = static_cast<int32_t>(a.t + 1);
            a.units[2] = 1;
        }
        s_retrieve = !reuse;
    }
    __syncthreads();
    if (s_retrieve)
        for (int i = threadIdx.x; i < D; i += blockDim.x) a.anchor[i] = __bfloat162float(q[i]);
}

// z[h][c] = sigma * q^(h) . k_c^(h / g) for the candidates c of this CTA's
// chunk [lo + chunk * blockIdx.x, + chunk): one thread per key, streaming its
// K row in 16-byte pieces (the query, in shared memory, is read as
// broadcasts). The chunk's logits are staged in shared memory, written out as
// whole rows, and summarised per head as (max, sum of exp(z - max)).
__global__ void __launch_bounds__(128) k_dec_logits(DecArgs a, const __nv_bfloat16* __restrict__ q,
                                                    const uint4* __restrict__ k)
{
    if (!a.state[2]) return;
    extern __shared__ float sm[];
    float* qs = sm;                        // [H_q][128]
    float* zs = sm + a.Hq * kHeadDim;      // [H_q][chunk]
    const int D = a.Hq * kHeadDim;
    for (int i = threadIdx.x; i < D; i += blockDim.x) qs[i] = __bfloat162float(q[i]);
    __syncthreads();
    const int64_t lo = a.n_sink, hi = window_start(a, a.t);
    const int64_t c0 = lo + static_cast<int64_t>(blockIdx.x) * a.chunk;
    const int n = static_cast<int>((hi - c0 < a.chunk) ? hi - c0 : a.chunk);
    const int i = threadIdx.x;
    if (i < n) {
        const int64_t c = c0 + i;
        for (int j = 0; j < a.Hkv; ++j) {
            const uint4* kr = k + (c * a.Hkv + j) * 16;  // 16 pieces of 8 bf16
            uint4 kv[16];
#pragma unroll
            for (int p = 0; p < 16; ++p) kv[p] = kr[p];
            for (int hl = 0; hl < a.g; ++hl) {
                const float4* qh = reinterpret_cast<const float4*>(qs + (j * a.g + hl) * kHeadDim);
                float acc = 0.f;
#pragma unroll
                for (int p = 0; p < 16; ++p) {
                    const float4 qa = qh[2 * p], qb = qh[2 * p + 1];
                    acc += qa.x * bf16_lo(kv[p].x) + qa.y * bf16_hi(kv[p].x) + qa.z * bf16_lo(kv[p].y) +
                           qa.w * bf16_hi(kv[p].y) + qb.x * bf16_lo(kv[p].z) + qb.y * bf16_hi(kv[p].z) +
                           qb.z * bf16_lo(kv[p].w) + qb.w * bf16_hi(kv[p].w);
                }
                zs[(j * a.g + hl) * a.chunk + i] = a.sigma * acc;
            }
        }
    }
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int h = warp; h < a.Hq; h += blockDim.x / 32) {
        const float* zh = zs + h * a.chunk;
        float* dst = a.z + h * a.cap + c0;
        float m = -INFINITY;
        for (int ii = lane; ii < n; ii += 32) {
            dst[ii] = zh[ii];
            m = fmaxf(m, zh[ii]);
        }
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
        float sum = 0.f;
        for (int ii = lane; ii < n; ii += 32) sum += expf(zh[ii] - m);
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
        if (lane == 0) a.zpart[static_cast<int64_t>(blockIdx.x) * a.Hq + h] = make_float2(m, sum);
    }
}

// Per head (one warp): the chunks' (max, sum) merged into max and 1 / sum.
__global__ void __launch_bounds__(256) k_dec_stats(DecArgs a, int n_chunks)
{
    if (!a.state[2]) return;
    const int h = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (h >= a.Hq) return;
    float m = -INFINITY;
    for (int b = lane; b < n_chunks; b += 32) m = fmaxf(m, a.zpart[static_cast<int64_t>(b) * a.Hq + h].x);
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    float s = 0.f;
    for (int b = lane; b < n_chunks; b += 32) {
        const float2 p = a.zpart[static_cast<int64_t>(b) * a.Hq + h];
        if (p.x > -INFINITY) s += p.y * expf(p.x - m);
    }
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
    if (lane == 0) a.stats[h] = make_float2(m, s > 0.f ? 1.0f / s : 0.f);
}

// score[c] = sum over heads (in order) of exp(z - max) / sum; NaN off the candidates.
__global__ void __launch_bounds__(256) k_dec_vote(DecArgs a)
{
    if (!a.state[2]) return;
    const int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (c > a.t) return;
    const int64_t lo = a.n_sink, hi = window_start(a, a.t);
    float sc = __int_as_float(0x7FC00000);
    if (c >= lo && c < hi) {
        sc = 0.f;
        for (int h = 0; h < a.Hq; ++h) {
            const float2 st = a.stats[h];
            sc += expf(a.z[h * a.cap + c] - st.x) * st.y;
        }
    }
    a.scores[c] = sc;
}

// Attention of the query over its keys, split over key chunks (blockIdx.y):
// key i of the step is the sink i (i < n_s = min(n_sink, W_t)), then the
// cached selection (produced by the top-k: ascending, inside [n_sink, W_a)
// with W_a <= W_t), then the window [W_t, t]. One warp per query head of KV
// head blockIdx.x, lane l holding dimensions [4 l, 4 l + 4); online softmax in
// log2 units. Writes (max, sum, unnormalised o) per (head, split).
__global__ void __launch_bounds__(256) k_dec_attn(DecArgs a, const __nv_bfloat16* __restrict__ q,
                                                  const uint2* __restrict__ k, const uint2* __restrict__ v)
{
    const int j = blockIdx.x, split = blockIdx.y;
    const int lane = threadIdx.x & 31, hl = threadIdx.x >> 5;
    if (hl >= a.g) return;
    const int h = j * a.g + hl;
    const int64_t W = window_start(a, a.t);
    const int n_s = static_cast<int>(a.n_sink < W ? a.n_sink : W);
    int n_sel = *a.sel_count;
    n_sel = n_sel < 0 ? 0 : (n_sel > a.k ? a.k : n_sel);
    const int n = n_s + n_sel + static_cast<int>(a.t - W + 1);
    const int per = (n + a.splits - 1) / a.splits;
    const int i0 = split * per, i1 = (i0 + per < n) ? i0 + per : n;
    const __nv_bfloat16* qh = q + h * kHeadDim + 4 * lane;
    const float q0 = __bfloat162float(qh[0]), q1 = __bfloat162float(qh[1]);
    const float q2 = __bfloat162float(qh[2]), q3 = __bfloat162float(qh[3]);
    float m = -INFINITY, l = 0.f, o0 = 0.f, o1 = 0.f, o2 = 0.f, o3 = 0.f;
#pragma unroll 4
    for (int i = i0; i < i1; ++i) {
        const int64_t tok = i < n_s ? i : (i < n_s + n_sel ? a.sel[i - n_s] : W + (i - n_s - n_sel));
        const int64_t row = (tok * a.Hkv + j) * 32 + lane;
        const uint2 kw = k[row];
        const uint2 vw = v[row];
        float s = q0 * bf16_lo(kw.x) + q1 * bf16_hi(kw.x) + q2 * bf16_lo(kw.y) + q3 * bf16_hi(kw.y);
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
        s *= a.attn_scale_log2;
        const float m_new = fmaxf(m, s);
        const float alpha = exp2f(m - m_new), p = exp2f(s - m_new);
        l = l * alpha + p;
        o0 = o0 * alpha + p * bf16_lo(vw.x);
        o1 = o1 * alpha + p * bf16_hi(vw.x);
        o2 = o2 * alpha + p * bf16_lo(vw.y);
        o3 = o3 * alpha + p * bf16_hi(vw.y);
        m = m_new;
    }
    float* pt = a.part + (static_cast<int64_t>(h) * a.splits + split) * 130;
    if (lane == 0) {
        pt[0] = m;
        pt[1] = l;
    }
    pt[2 + 4 * lane] = o0;
    pt[3 + 4 * lane] = o1;
    pt[4 + 4 * lane] = o2;
    pt[5 + 4 * lane] = o3;
}

// Merge the splits of every head (in order) and write the bf16 output row.
__global__ void __launch_bounds__(128) k_dec_combine(DecArgs a, __nv_bfloat16* __restrict__ out)
{
    const int h = blockIdx.x, d = threadIdx.x;
    const float* ph = a.part + static_cast<int64_t>(h) * a.splits * 130;
    float m = -INFINITY;
    for (int s = 0; s < a.splits; ++s) m = fmaxf(m, ph[s * 130]);
    float l = 0.f, o = 0.f;
    for (int s = 0; s < a.splits; ++s) {
        const float ms = ph[s * 130];
        if (ms == -INFINITY) continue;
        const float w = exp2f(ms - m);
        l += ph[s * 130 + 1] * w;
        o += ph[s * 130 + 2 + d] * w;
    }
    out[h * kHeadDim + d] = __float2bfloat16_rn(l > 0.f ? o / l : 0.f);
}

}  // namespace

size_t decode_cache_bytes(const Derived& d)
{
    return kDecAnchor + static_cast<size_t>(d.Hq) * kHeadDim * sizeof(float) +
           static_cast<size_t>(d.k > 0 ? d.k : 1) * sizeof(int32_t) + 256;
}

size_t decode_ws_bytes(const Derived& d, int splits)
{
    const size_t cap = static_cast<size_t>(d.N);
    size_t off = 0;
    off = align_up(off + 256, kAlign);                                           // status word
    off = align_up(off + static_cast<size_t>(d.Hq) * cap * sizeof(float), kAlign);  // z
    off = align_up(off + static_cast<size_t>(d.Hq) * sizeof(float2), kAlign);   // stats
    off = align_up(off + cap * sizeof(float), kAlign);                          // scores
    off = align_up(off + static_cast<size_t>(d.Hq) * splits * 130 * sizeof(float), kAlign);
    off = align_up(off + static_cast<size_t>(d.Hq) * ((cap + 127) / 128) * sizeof(float2), kAlign);  // zpart
    off = align_up(off + (256 + 4) * sizeof(int32_t), kAlign);                                    // top-k hist, state
    off = align_up(off + static_cast<size_t>(topk_max_chunks(d)) * sizeof(int2), kAlign);          // top-k counts
    return off;
}

constexpr int kDecSplits = 128;

int decode_splits() { return kDecSplits; }

cudaError_t launch_decode_step(const Derived& d, int64_t t, const void* q, const void* k, const void* v,
                               uint8_t* cache, void* out, uint8_t* ws, cudaStream_t st)
{
    DecArgs a;
    a.Hq = d.Hq;
    a.Hkv = d.Hkv;
    a.g = d.g;
    a.t = t;
    a.cap = d.N;
    a.n_sink = d.n_sink;
    a.n_local = d.n_local;
    a.k = d.k;
    a.S_max = d.S_max;
    a.theta = d.theta;
    a.sigma = d.sigma;
    a.attn_scale_log2 = d.attn_scale * 1.4426950408889634f;
    a.state = reinterpret_cast<int32_t*>(cache + kDecState);
    a.units = reinterpret_cast<int32_t*>(cache + kDecUnits);
    a.anchor = reinterpret_cast<float*>(cache + kDecAnchor);
    a.sel = reinterpret_cast<int32_t*>(cache + kDecAnchor + static_cast<size_t>(d.Hq) * kHeadDim * sizeof(float));
    a.sel_count = a.sel + (d.k > 0 ? d.k : 1);
    a.splits = kDecSplits;
    size_t off = 256;
    auto take = [&](size_t bytes) {
        const size_t at = off;
        off = align_up(off + bytes, kAlign);
        return at;
    };
    const size_t cap = static_cast<size_t>(d.N);
    a.z = reinterpret_cast<float*>(ws + take(static_cast<size_t>(d.Hq) * cap * sizeof(float)));
    a.stats = reinterpret_cast<float2*>(ws + take(static_cast<size_t>(d.Hq) * sizeof(float2)));
    a.scores = reinterpret_cast<float*>(ws + take(cap * sizeof(float)));
    a.part = reinterpret_cast<float*>(ws + take(static_cast<size_t>(d.Hq) * kDecSplits * 130 * sizeof(float)));
    a.zpart = reinterpret_cast<float2*>(ws + take(static_cast<size_t>(d.Hq) * ((cap + 127) / 128) * sizeof(float2)));
    a.chunk = 128;  // 32 KB of staged logits for 32 heads: several CTAs per SM keep loads in flight
    int32_t* tk_hist = reinterpret_cast<int32_t*>(ws + take((256 + 4) * sizeof(int32_t)));
    int2* tk_counts = reinterpret_cast<int2*>(ws + take(static_cast<size_t>(topk_max_chunks(d)) * sizeof(int2)));

    const auto* qb = static_cast<const __nv_bfloat16*>(q);
    k_dec_gate<<<1, 256, 0, st>>>(a, qb);
    const int64_t n_cand = window_start(a, t) - d.n_sink;
    if (n_cand > 0) {
        const int n_chunks = static_cast<int>((n_cand + a.chunk - 1) / a.chunk);
        const size_t smem = (static_cast<size_t>(d.Hq) * kHeadDim + static_cast<size_t>(d.Hq) * a.chunk) * sizeof(float);
        cudaError_t e0 = cudaFuncSetAttribute(k_dec_logits, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              static_cast<int>(smem));
        if (e0 != cudaSuccess) return e0;
        k_dec_logits<<<n_chunks, 128, smem, st>>>(a, qb, static_cast<const uint4*>(k));
        k_dec_stats<<<(d.Hq + 7) / 8, 256, 0, st>>>(a, n_chunks);
        k_dec_vote<<<static_cast<unsigned>((t + 1 + 255) / 256), 256, 0, st>>>(a);
        // top-k of the one-unit table [t, t + 1] kept in the cache, gated on the retrieval flag
        Derived du = d;
        du.L = 1;
        du.B = 1;
        du.nb = d.N;
        const Units ut{a.units, a.units + 2, 0, d.N, 1, static_cast<int>(d.N)};
        const TopkScratch scratch{tk_hist, tk_hist + 256, tk_counts, topk_max_chunks(du)};
        cudaError_t e = launch_topk(du, ut, static_cast<int>(t), static_cast<int>(t + 1), a.scores, a.sel,
                                    a.sel_count, st, a.state + 2, &scratch);
        if (e != cudaSuccess) return e;
    } else {
        // no candidates: the selection is empty whenever this step retrieves
        cudaError_t e = cudaMemsetAsync(a.sel_count, 0, sizeof(int32_t), st);
        if (e != cudaSuccess) return e;
    }
    k_dec_attn<<<dim3(d.Hkv, kDecSplits), 32 * d.g, 0, st>>>(a, qb, static_cast<const uint2*>(k),
                                                              static_cast<const uint2*>(v));
    k_dec_combine<<<d.Hq, kHeadDim, 0, st>>>(a, static_cast<__nv_bfloat16*>(out));
    return cudaGetLastError();
}

}  // namespace scale
