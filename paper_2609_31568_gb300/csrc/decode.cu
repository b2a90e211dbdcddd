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
    int32_t* list;      // distant + window keys of this step
    int32_t* list_n;
    float* part;        // [H_q][splits][130]: max, sum, o[128]
    int splits;
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

// z[h][c] = sigma * q^(h) . k_c^(h / g) for the candidates c; one warp per key,
// lane l holding dimensions [4 l, 4 l + 4) of every head.
__global__ void __launch_bounds__(256) k_dec_logits(DecArgs a, const __nv_bfloat16* __restrict__ q,
                                                    const uint2* __restrict__ k)
{
    if (!a.state[2]) return;
    extern __shared__ float qs[];  // [H_q][128]
    const int D = a.Hq * kHeadDim;
    for (int i = threadIdx.x; i < D; i += blockDim.x) qs[i] = __bfloat162float(q[i]);
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t lo = a.n_sink, hi = window_start(a, a.t);
    for (int64_t c = lo + static_cast<int64_t>(blockIdx.x) * 8 + warp; c < hi; c += static_cast<int64_t>(gridDim.x) * 8) {
        for (int j = 0; j < a.Hkv; ++j) {
            const uint2 kw = k[(c * a.Hkv + j) * 32 + lane];  // 4 bf16 of this lane
            const float k0 = bf16_lo(kw.x), k1 = bf16_hi(kw.x), k2 = bf16_lo(kw.y), k3 = bf16_hi(kw.y);
            for (int hl = 0; hl < a.g; ++hl) {
                const int h = j * a.g + hl;
                const float* qh = qs + h * kHeadDim + 4 * lane;
                float d = qh[0] * k0 + qh[1] * k1 + qh[2] * k2 + qh[3] * k3;
                for (int o = 16; o > 0; o >>= 1) d += __shfl_xor_sync(0xFFFFFFFFu, d, o);
                if (lane == 0) a.z[h * a.cap + c] = a.sigma * d;
            }
        }
    }
}

// Per head: max of z over the candidates and 1 / sum of exp(z - max).
__global__ void __launch_bounds__(256) k_dec_stats(DecArgs a)
{
    if (!a.state[2]) return;
    __shared__ float red[8];
    const int h = blockIdx.x;
    const int64_t lo = a.n_sink, hi = window_start(a, a.t);
    const float* zh = a.z + h * a.cap;
    float m = -INFINITY;
    for (int64_t c = lo + threadIdx.x; c < hi; c += blockDim.x) m = fmaxf(m, zh[c]);
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
    __syncthreads();
    m = red[0];
    for (int i = 1; i < 8; ++i) m = fmaxf(m, red[i]);
    __syncthreads();
    float s = 0.f;
    for (int64_t c = lo + threadIdx.x; c < hi; c += blockDim.x) s += expf(zh[c] - m);
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.f;
        for (int i = 0; i < 8; ++i) t += red[i];
        a.stats[h] = make_float2(m, t > 0.f ? 1.0f / t : 0.f);
    }
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

// Key list of the step (one warp): sinks [0, min(n_sink, W_t)), the cached
// selection's valid entries (inside [n_sink, W_t), increasing), the window [W_t, t].
__global__ void __launch_bounds__(32) k_dec_list(DecArgs a)
{
    const int lane = threadIdx.x;
    const int64_t W = window_start(a, a.t);
    const int n_s = static_cast<int>(a.n_sink < W ? a.n_sink : W);
    for (int i = lane; i < n_s; i += 32) a.list[i] = i;
    int base = n_s;
    int cnt = *a.sel_count;
    cnt = cnt < 0 ? 0 : (cnt > a.k ? a.k : cnt);
    for (int c0 = 0; c0 < cnt; c0 += 32) {
        const int i = c0 + lane;
        bool valid = false;
        int32_t tok = 0;
        if (i < cnt) {
            tok = a.sel[i];
            valid = tok >= a.n_sink && tok < W && (i == 0 || tok > a.sel[i - 1]);
        }
        const uint32_t b = __ballot_sync(0xFFFFFFFFu, valid);
        if (valid) a.list[base + __popc(b & ((1u << lane) - 1u))] = tok;
        base += __popc(b);
    }
    const int n_w = static_cast<int>(a.t - W + 1);
    for (int i = lane; i < n_w; i += 32) a.list[base + i] = static_cast<int32_t>(W + i);
    if (lane == 0) *a.list_n = base + n_w;
}

// Attention of the query over the listed keys, split over key chunks
// (blockIdx.y): one warp per query head of KV head blockIdx.x, lane l holding
// dimensions [4 l, 4 l + 4); online softmax in log2 units. Writes (max, sum,
// unnormalised o) per (head, split).
__global__ void __launch_bounds__(256) k_dec_attn(DecArgs a, const __nv_bfloat16* __restrict__ q,
                                                  const uint2* __restrict__ k, const uint2* __restrict__ v)
{
    const int j = blockIdx.x, split = blockIdx.y;
    const int lane = threadIdx.x & 31, hl = threadIdx.x >> 5;
    if (hl >= a.g) return;
    const int h = j * a.g + hl;
    const int n = *a.list_n;
    const int per = (n + a.splits - 1) / a.splits;
    const int i0 = split * per, i1 = (i0 + per < n) ? i0 + per : n;
    const __nv_bfloat16* qh = q + h * kHeadDim + 4 * lane;
    const float q0 = __bfloat162float(qh[0]), q1 = __bfloat162float(qh[1]);
    const float q2 = __bfloat162float(qh[2]), q3 = __bfloat162float(qh[3]);
    float m = -INFINITY, l = 0.f, o0 = 0.f, o1 = 0.f, o2 = 0.f, o3 = 0.f;
#pragma unroll 4
    for (int i = i0; i < i1; ++i) {
        const int64_t row = (static_cast<int64_t>(a.list[i]) * a.Hkv + j) * 32 + lane;
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
    off = align_up(off + (static_cast<size_t>(d.n_sink) + d.k + d.n_local + 1) * sizeof(int32_t) + 16, kAlign);
    off = align_up(off + static_cast<size_t>(d.Hq) * splits * 130 * sizeof(float), kAlign);
    return off;
}

constexpr int kDecSplits = 64;

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
    a.list = reinterpret_cast<int32_t*>(ws + take((static_cast<size_t>(d.n_sink) + d.k + d.n_local + 1) * sizeof(int32_t) + 16));
    a.list_n = a.list + d.n_sink + d.k + d.n_local + 1;
    a.part = reinterpret_cast<float*>(ws + take(static_cast<size_t>(d.Hq) * kDecSplits * 130 * sizeof(float)));

    const auto* qb = static_cast<const __nv_bfloat16*>(q);
    k_dec_gate<<<1, 256, 0, st>>>(a, qb);
    const int64_t n_cand = window_start(a, t) - d.n_sink;
    if (n_cand > 0) {
        const unsigned blocks = static_cast<unsigned>(std::min<int64_t>((n_cand + 7) / 8, 152 * 16));
        const size_t qsm = static_cast<size_t>(d.Hq) * kHeadDim * sizeof(float);
        k_dec_logits<<<blocks, 256, qsm, st>>>(a, qb, static_cast<const uint2*>(k));
        k_dec_stats<<<d.Hq, 256, 0, st>>>(a);
        k_dec_vote<<<static_cast<unsigned>((t + 1 + 255) / 256), 256, 0, st>>>(a);
        // top-k of the one-unit table [t, t + 1] kept in the cache, gated on the retrieval flag
        Derived du = d;
        du.L = 1;
        du.B = 1;
        du.nb = d.N;
        const Units ut{a.units, a.units + 2, 0, d.N, 1, static_cast<int>(d.N)};
        cudaError_t e = launch_topk(du, ut, static_cast<int>(t), static_cast<int>(t + 1), a.scores, a.sel,
                                    a.sel_count, st, a.state + 2);
        if (e != cudaSuccess) return e;
    } else {
        // no candidates: the selection is empty whenever this step retrieves
        cudaError_t e = cudaMemsetAsync(a.sel_count, 0, sizeof(int32_t), st);
        if (e != cudaSuccess) return e;
    }
    k_dec_list<<<1, 32, 0, st>>>(a);
    k_dec_attn<<<dim3(d.Hkv, kDecSplits), 32 * d.g, 0, st>>>(a, qb, static_cast<const uint2*>(k),
                                                              static_cast<const uint2*>(v));
    k_dec_combine<<<d.Hq, kHeadDim, 0, st>>>(a, static_cast<__nv_bfloat16*>(out));
    return cudaGetLastError();
}

}  // namespace scale
