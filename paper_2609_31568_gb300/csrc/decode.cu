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
// Scoring one query against every key is a matrix-vector product per KV head,
// bound by reading K once: k_dec_logits_tc streams the keys by TMA and runs
// the products on the tensor cores; shapes it does not cover use CUDA-core
// kernels. Whether the step retrieves is decided on the device, so a step
// never synchronises with the host.
#include <cuda_bf16.h>

#include <cmath>

#include "ptx_sm103.cuh"
#include "scale_internal.h"
#include "tma_host.h"

namespace scale {
namespace {

using namespace scale_ptx;

// Decode cache layout (bytes from its base).
constexpr size_t kDecState = 0;     // int32[8]: valid, steps, retrieve, -, anchor position
constexpr size_t kDecUnits = 64;    // int32[2] unit table [t, t + 1] of the anchor, int32 n_units
constexpr size_t kDecAnchor = 256;  // fp32 [H_q * 128]
// selection int32 [k] and its count follow the anchor

// Read-only 16-byte load; volatile keeps a run of them issued back to back.
__device__ __forceinline__ uint4 ld_nc(const uint4* p)
{
    uint4 r;
    asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

constexpr int kDecSplits = 128;

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
    float2* zpart;      // [H_q][n_stat] (max, sum) of each candidate chunk
    int n_stat;         // candidate chunks (64 keys, or 128 for the tensor-core logits)
    int32_t* status;    // device status word of the workspace
    uint64_t timeout_ns;
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

// Merge of two (max, sum of exp(z - max)) summaries; symmetric in its
// arguments, so both lanes of a butterfly get the same bits.
__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2)
{
    const float mn = fmaxf(m, m2);
    s = (m == -INFINITY ? 0.f : s * expf(m - mn)) + (m2 == -INFINITY ? 0.f : s2 * expf(m2 - mn));
    m = mn;
}

// z[h][c] = sigma * q^(h) . k_c^(h / g) for the candidates c in
// [n_sink, W_t), G = g query heads per KV head. A CTA takes 512 candidates,
// warp w the 64 from c0 + 64 w: lane l the four keys c0 + 64 w + l / 2 + 16 r
// (r < 4) and the 16-byte pieces l % 2, l % 2 + 2, ... of each key's 256-byte
// row for KV head j, so each load instruction reads 16 keys x one whole
// 32-byte sector. A query piece read from shared memory feeds the four keys
// (shared-memory traffic per key is a quarter of one key per thread), every
// key piece is unpacked once for the G heads, one shuffle joins the halves.
// Each warp writes its logits straight to z and summarises every head over
// its 64 keys as (max, sum of exp(z - max)) in zpart[h][chunk], chunk =
// 8 blockIdx.x + w, merged across lanes by a fixed butterfly.
constexpr int kDecStat = 64;         // candidates per (max, sum) summary
constexpr int kDecBlockKeys = 512;   // candidates per CTA of k_dec_logits

template <int G>
__global__ void __launch_bounds__(256) k_dec_logits(DecArgs a, const __nv_bfloat16* __restrict__ q,
                                                    const uint4* __restrict__ k)
{
    if (!a.state[2]) return;
    extern __shared__ float qs[];  // [H_q][128]
    const int D = a.Hq * kHeadDim;
    for (int i = threadIdx.x; i < D; i += blockDim.x) qs[i] = __bfloat162float(q[i]);
    __syncthreads();
    const int64_t lo = a.n_sink, hi = window_start(a, a.t);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, half = lane & 1;
    const int64_t cw = lo + static_cast<int64_t>(blockIdx.x) * kDecBlockKeys + kDecStat * warp;
    if (cw >= hi) return;  // warp-uniform; no barrier follows
    const int64_t cl = cw + (lane >> 1);
    const int64_t chunk = static_cast<int64_t>(blockIdx.x) * (kDecBlockKeys / kDecStat) + warp;
    bool live[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) live[r] = cl + 16 * r < hi;
    const uint4 zero = make_uint4(0, 0, 0, 0);
    constexpr int UU = G <= 4 ? 2 : 1;  // pieces per key in flight together (registers)
    for (int j = 0; j < a.Hkv; ++j) {
        float acc[4][G];
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
            for (int hl = 0; hl < G; ++hl) acc[r][hl] = 0.f;
        const uint4* kr = k + (cl * a.Hkv + j) * 16 + half;
        const int64_t key_step = static_cast<int64_t>(16) * a.Hkv * 16;  // 16 keys, in uint4
        const float* qj = qs + j * G * kHeadDim + 8 * half;
#pragma unroll
        for (int u0 = 0; u0 < 8; u0 += UU) {
            uint4 kv[UU][4];
#pragma unroll
            for (int uu = 0; uu < UU; ++uu)
#pragma unroll
                for (int r = 0; r < 4; ++r)
                    kv[uu][r] = live[r] ? ld_nc(kr + r * key_step + 2 * (u0 + uu)) : zero;
#pragma unroll
            for (int uu = 0; uu < UU; ++uu) {
                float4 qa[G], qb[G];
#pragma unroll
                for (int hl = 0; hl < G; ++hl) {
                    const float4* qh = reinterpret_cast<const float4*>(qj + hl * kHeadDim + 16 * (u0 + uu));
                    qa[hl] = qh[0];
                    qb[hl] = qh[1];
                }
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    const uint4 w = kv[uu][r];
                    const float x0 = bf16_lo(w.x), x1 = bf16_hi(w.x), x2 = bf16_lo(w.y), x3 = bf16_hi(w.y);
                    const float x4 = bf16_lo(w.z), x5 = bf16_hi(w.z), x6 = bf16_lo(w.w), x7 = bf16_hi(w.w);
#pragma unroll
                    for (int hl = 0; hl < G; ++hl)
                        acc[r][hl] += qa[hl].x * x0 + qa[hl].y * x1 + qa[hl].z * x2 + qa[hl].w * x3 +
                                      qb[hl].x * x4 + qb[hl].y * x5 + qb[hl].z * x6 + qb[hl].w * x7;
                }
            }
        }
#pragma unroll
        for (int hl = 0; hl < G; ++hl) {
            const int h = j * G + hl;
            float zv[4];
#pragma unroll
            for (int r = 0; r < 4; ++r) zv[r] = a.sigma * (acc[r][hl] + __shfl_xor_sync(0xFFFFFFFFu, acc[r][hl], 1));
            float* zh = a.z + static_cast<int64_t>(h) * a.cap;
#pragma unroll
            for (int r = 0; r < 4; ++r)
                if ((r >> 1) == half && live[r]) zh[cl + 16 * r] = zv[r];  // half 0: keys 0, 1; half 1: 2, 3
            float m = -INFINITY;
#pragma unroll
            for (int r = 0; r < 4; ++r)
                if (live[r]) m = fmaxf(m, zv[r]);
            float sum = 0.f;
#pragma unroll
            for (int r = 0; r < 4; ++r)
                if (live[r]) sum += expf(zv[r] - m);
            for (int o = 2; o < 32; o <<= 1)  // the two lanes of a key hold the same values
                merge_ms(m, sum, __shfl_xor_sync(0xFFFFFFFFu, m, o), __shfl_xor_sync(0xFFFFFFFFu, sum, o));
            if (lane == 0) a.zpart[static_cast<int64_t>(h) * a.n_stat + chunk] = make_float2(m, sum);
        }
    }
}

// Any group size: two lanes per key (every other 16-byte piece of its row),
// the query heads of the KV head looped at run time; 128 candidates per CTA,
// logits staged in shared memory and summarised per 64 keys as above.
__global__ void __launch_bounds__(256) k_dec_logits_any(DecArgs a, const __nv_bfloat16* __restrict__ q,
                                                        const uint4* __restrict__ k)
{
    if (!a.state[2]) return;
    extern __shared__ float sm[];
    float* qs = sm;                        // [H_q][128]
    float* zs = sm + a.Hq * kHeadDim;      // [H_q][128]
    const int D = a.Hq * kHeadDim;
    for (int i = threadIdx.x; i < D; i += blockDim.x) qs[i] = __bfloat162float(q[i]);
    __syncthreads();
    const int64_t lo = a.n_sink, hi = window_start(a, a.t);
    const int64_t c0 = lo + static_cast<int64_t>(blockIdx.x) * 128;
    const int n = static_cast<int>((hi - c0 < 128) ? hi - c0 : 128);
    const int i = threadIdx.x >> 1, half = threadIdx.x & 1;
    const bool live = i < n;
    const uint4 zero = make_uint4(0, 0, 0, 0);
    for (int j = 0; j < a.Hkv; ++j) {
        const uint4* kr = k + ((c0 + i) * a.Hkv + j) * 16 + half;
        uint4 kv[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) kv[u] = live ? ld_nc(kr + 2 * u) : zero;
        for (int hl = 0; hl < a.g; ++hl) {
            const float4* qh = reinterpret_cast<const float4*>(qs + (j * a.g + hl) * kHeadDim + 8 * half);
            float acc = 0.f;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const float4 qa = qh[4 * u], qb = qh[4 * u + 1];
                acc += qa.x * bf16_lo(kv[u].x) + qa.y * bf16_hi(kv[u].x) + qa.z * bf16_lo(kv[u].y) +
                       qa.w * bf16_hi(kv[u].y) + qb.x * bf16_lo(kv[u].z) + qb.y * bf16_hi(kv[u].z) +
                       qb.z * bf16_lo(kv[u].w) + qb.w * bf16_hi(kv[u].w);
            }
            acc += __shfl_xor_sync(0xFFFFFFFFu, acc, 1);
            if (live && !half) zs[(j * a.g + hl) * 128 + i] = a.sigma * acc;
        }
    }
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int hs = warp; hs < 2 * a.Hq; hs += blockDim.x / 32) {
        const int h = hs >> 1, sub = hs & 1;
        const int b0 = sub * kDecStat, b1 = n < b0 + kDecStat ? n : b0 + kDecStat;
        if (b1 <= b0) continue;  // past the candidates: never read
        const float* zh = zs + h * 128;
        float* dst = a.z + static_cast<int64_t>(h) * a.cap + c0;
        float m = -INFINITY;
        for (int ii = b0 + lane; ii < b1; ii += 32) {
            dst[ii] = zh[ii];
            m = fmaxf(m, zh[ii]);
        }
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
        float sum = 0.f;
        for (int ii = b0 + lane; ii < b1; ii += 32) sum += expf(zh[ii] - m);
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
        if (lane == 0) a.zpart[static_cast<int64_t>(h) * a.n_stat + blockIdx.x * 2 + sub] = make_float2(m, sum);
    }
}

// Tensor-core form of the logits (g <= 16 query heads per KV head, H_kv <=
// 16): a persistent CTA per SM walks its share of the items (128-key tile,
// KV head j). Warp 0 lane 0 streams the tile's keys of head j by TMA (two
// 64-dimension boxes of 128 rows, 32 KB, 128-byte swizzle) into a 4-stage
// ring, so about 96 KB per SM are in flight without holding registers; warp 1
// lane 0 issues D[key][row] = K_j . Q_j^T as eight tcgen05.mma (M = 128 keys,
// N = 16: the g query rows of head j, then zero rows; K = 128) into one of two
// 16-column TMEM accumulators; warps 2-5 read their 32 keys' columns, write
// z = sigma * D for the live keys (W_t and beyond are dropped) and merge
// each head's (max, sum of exp(z - max)) over the tile: a butterfly inside the
// warp, then the four warps in TMEM-lane order. The query operand is written
// to shared memory by the threads in the swizzled K-major layout the MMA
// reads. Every wait is bounded; on expiry the kernel records
// SCALE_ERR_TIMEOUT, drains what it issued and frees its TMEM.
constexpr int kDtStages = 4;
constexpr uint32_t kDtTile = 128 * 128 * 2;  // 128 keys x 128 dims (two 64-dim halves)
constexpr uint32_t kDtHalf = kDtTile / 2;
constexpr uint32_t kDtQ = 16 * 128 * 2;      // query rows of one KV head
constexpr uint32_t kDtQHalf = kDtQ / 2;
constexpr int kDtMaxHkv = 16;
constexpr uint32_t kDtSmem = kDtStages * kDtTile + kDtMaxHkv * kDtQ + 1024;
constexpr int kDtThreads = 192;
static_assert(kDtSmem <= 227 * 1024 - 1024, "tensor-core decode logits shared memory");

struct DtBars {
    uint64_t k_full[kDtStages], k_empty[kDtStages];
    uint64_t d_full[2], d_empty[2];
    uint64_t drain;
};

__device__ __forceinline__ void dt_fail(volatile int* abort_flag, int32_t* status)
{
    *abort_flag = 1;
    record_status(status, SCALE_ERR_TIMEOUT);
}

template <int G>
__global__ void __launch_bounds__(kDtThreads, 1)
k_dec_logits_tc(const __grid_constant__ CUtensorMap tk, const DecArgs a, const __nv_bfloat16* __restrict__ q)
{
    if (!a.state[2]) return;
    extern __shared__ uint8_t smem_raw[];
    __shared__ DtBars bars;
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    __shared__ float2 s_stat[2][4][G];
    const int64_t lo = a.n_sink, hi = window_start(a, a.t);
    const int64_t items = (hi - lo + 127) / 128 * a.Hkv;
    const int64_t i0 = items * blockIdx.x / gridDim.x, i1 = items * (blockIdx.x + 1) / gridDim.x;
    if (i1 <= i0) return;
    const int n_it = static_cast<int>(i1 - i0);
    uint8_t* smem = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
    uint8_t* kbuf = smem;
    uint8_t* qbuf = smem + kDtStages * kDtTile;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    // query operand: row r of head j is query head j G + r (zero for r >= G);
    // 16-byte chunk c of a 128-byte row goes to chunk c ^ (row % 8)
    for (int x = tid; x < a.Hkv * 16 * 16; x += blockDim.x) {
        const int c = x & 15, r = (x >> 4) & 15, j = x >> 8;
        uint4 val = make_uint4(0, 0, 0, 0);
        if (r < G) val = *reinterpret_cast<const uint4*>(q + (static_cast<int64_t>(j) * G + r) * kHeadDim + 8 * c);
        const int hf = c >> 3, cc = c & 7;
        *reinterpret_cast<uint4*>(qbuf + j * kDtQ + hf * kDtQHalf + (r >> 3) * 1024 + (r & 7) * 128 +
                                  ((cc ^ (r & 7)) << 4)) = val;
    }
    fence_proxy_async_smem();
    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < kDtStages; ++i) {
            mbar_init(&bars.k_full[i], 1);
            mbar_init(&bars.k_empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars.d_full[i], 1);
            mbar_init(&bars.d_empty[i], 128);
        }
        mbar_init(&bars.drain, 1);
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc(&tmem_slot, 32);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&tk);
            int issued[kDtStages] = {};
            for (int it = 0; it < n_it && !abort_flag; ++it) {
                const int st = it % kDtStages;
                if (it >= kDtStages &&
                    !mbar_wait_bounded(&bars.k_empty[st], ((it / kDtStages) - 1) & 1, a.timeout_ns, &abort_flag)) {
                    dt_fail(&abort_flag, a.status);
                    break;
                }
                const int64_t item = i0 + it;
                const int64_t tile = item / a.Hkv;
                const int j = static_cast<int>(item - tile * a.Hkv);
                const int32_t key0 = static_cast<int32_t>(lo + 128 * tile);
                mbar_arrive_expect_tx(&bars.k_full[st], kDtTile);
                ++issued[st];
                for (int hf = 0; hf < 2; ++hf)
                    tma_load_3d(kbuf + st * kDtTile + hf * kDtHalf, &tk, &bars.k_full[st], hf * 64, j, key0);
            }
            if (abort_flag)
                for (int st = 0; st < kDtStages; ++st)
                    if (issued[st]) mbar_wait_bounded(&bars.k_full[st], (issued[st] - 1) & 1, a.timeout_ns, nullptr);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, 16, 0);
            const uint64_t kdesc0 = sdesc_sw128(smem_addr(kbuf), 16, 1024);
            const uint64_t qdesc0 = sdesc_sw128(smem_addr(qbuf), 16, 1024);
            bool ok = true;
            for (int it = 0; it < n_it; ++it) {
                const int st = it % kDtStages, b = it & 1;
                if (!mbar_wait_bounded(&bars.k_full[st], (it / kDtStages) & 1, a.timeout_ns, &abort_flag)) {
                    ok = false;
                    break;
                }
                if (it >= 2 && !mbar_wait_bounded(&bars.d_empty[b], ((it >> 1) - 1) & 1, a.timeout_ns, &abort_flag)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int64_t item = i0 + it;
                const int j = static_cast<int>(item - item / a.Hkv * a.Hkv);
                mma_ss_k128_ab<kDtHalf, kDtQHalf>(tmem + b * 16, kdesc0 + st * (kDtTile >> 4),
                                                  qdesc0 + j * (kDtQ >> 4), idesc, 0u);
                mma_commit(&bars.d_full[b]);
                mma_commit(&bars.k_empty[st]);
            }
            if (!ok) {
                dt_fail(&abort_flag, a.status);
                mma_commit(&bars.drain);
                mbar_wait_bounded(&bars.drain, 0, a.timeout_ns, nullptr);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        // Every epilogue warp runs one named barrier per item, also after a
        // failed wait (it then skips the work).
        const int qq = warp & 3;  // TMEM lane quarter this warp may access
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(qq * 32) << 16);
        bool ok = true;
        for (int it = 0; it < n_it; ++it) {
            const int b = it & 1;
            const int64_t item = i0 + it;
            const int64_t tile = item / a.Hkv;
            const int j = static_cast<int>(item - tile * a.Hkv);
            if (ok) {
                ok = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(&bars.d_full[b], (it >> 1) & 1, a.timeout_ns, &abort_flag));
                if (ok) {
                    tc_fence_after();
                    uint32_t r[16];
                    tmem_ld16(lane_base + b * 16, r);
                    tmem_ld_wait();
                    tc_fence_before();
                    mbar_arrive(&bars.d_empty[b]);
                    const int64_t key = lo + 128 * tile + qq * 32 + lane;
                    const bool live = key < hi;
#pragma unroll
                    for (int hl = 0; hl < G; ++hl) {
                        const float zv = a.sigma * __uint_as_float(r[hl]);
                        if (live) a.z[static_cast<int64_t>(j * G + hl) * a.cap + key] = zv;
                        float m = live ? zv : -INFINITY, sum = live ? 1.f : 0.f;
                        for (int o = 1; o < 32; o <<= 1)
                            merge_ms(m, sum, __shfl_xor_sync(0xFFFFFFFFu, m, o), __shfl_xor_sync(0xFFFFFFFFu, sum, o));
                        if (lane == 0) s_stat[b][qq][hl] = make_float2(m, sum);
                    }
                }
            }
            named_barrier(1, 128);
            if (ok && qq == 0 && lane < G) {
                float2 t = s_stat[b][0][lane];
                for (int w = 1; w < 4; ++w) merge_ms(t.x, t.y, s_stat[b][w][lane].x, s_stat[b][w][lane].y);
                a.zpart[static_cast<int64_t>(j * G + lane) * a.n_stat + tile] = t;
            }
        }
        if (!ok) dt_fail(&abort_flag, a.status);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 32);
    }
}

// Fixed-order block reductions (warp butterflies, then the warps in order).
__device__ __forceinline__ float block_max256(float v, float* red)
{
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float m = red[0];
    for (int w = 1; w < static_cast<int>(blockDim.x >> 5); ++w) m = fmaxf(m, red[w]);
    __syncthreads();
    return m;
}

__device__ __forceinline__ float block_sum256(float v, float* red)
{
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float s = red[0];
    for (int w = 1; w < static_cast<int>(blockDim.x >> 5); ++w) s += red[w];
    __syncthreads();
    return s;
}

// Per head (one CTA of 256 threads): the chunks' (max, sum) merged into max
// and 1 / sum, thread t taking the chunks t, t + 256, ... in order.
__global__ void __launch_bounds__(256) k_dec_stats(DecArgs a, int n_chunks)
{
    if (!a.state[2]) return;
    __shared__ float red[8];
    const int h = blockIdx.x;
    const float2* zp = a.zpart + static_cast<int64_t>(h) * n_chunks;
    float m = -INFINITY;
    for (int b = threadIdx.x; b < n_chunks; b += blockDim.x) m = fmaxf(m, zp[b].x);
    m = block_max256(m, red);
    float s = 0.f;
    for (int b = threadIdx.x; b < n_chunks; b += blockDim.x) {
        const float2 p = zp[b];
        if (p.x > -INFINITY) s += p.y * expf(p.x - m);
    }
    s = block_sum256(s, red);
    if (threadIdx.x == 0) a.stats[h] = make_float2(m, s > 0.f ? 1.0f / s : 0.f);
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
// log2 units, eight keys per update (their loads and dot products are
// independent, so they overlap). Writes (max, sum, unnormalised o) per
// (head, split).
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
    auto key = [&](int i) -> int64_t {
        return i < n_s ? i : (i < n_s + n_sel ? a.sel[i - n_s] : W + (i - n_s - n_sel));
    };
    constexpr int KB = 8;  // keys per update
    int i = i0;
    for (; i + KB <= i1; i += KB) {
        uint2 kw[KB], vw[KB];
#pragma unroll
        for (int u = 0; u < KB; ++u) {
            const int64_t row = (key(i + u) * a.Hkv + j) * 32 + lane;
            kw[u] = k[row];
            vw[u] = v[row];
        }
        float s[KB];
#pragma unroll
        for (int u = 0; u < KB; ++u)
            s[u] = q0 * bf16_lo(kw[u].x) + q1 * bf16_hi(kw[u].x) + q2 * bf16_lo(kw[u].y) + q3 * bf16_hi(kw[u].y);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1)
#pragma unroll
            for (int u = 0; u < KB; ++u) s[u] += __shfl_xor_sync(0xFFFFFFFFu, s[u], o);
        float m_new = m;
#pragma unroll
        for (int u = 0; u < KB; ++u) {
            s[u] *= a.attn_scale_log2;
            m_new = fmaxf(m_new, s[u]);
        }
        const float alpha = exp2f(m - m_new);
        float p[KB], psum = 0.f;
#pragma unroll
        for (int u = 0; u < KB; ++u) {
            p[u] = exp2f(s[u] - m_new);
            psum += p[u];
        }
        l = l * alpha + psum;
        float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
#pragma unroll
        for (int u = 0; u < KB; ++u) {
            d0 += p[u] * bf16_lo(vw[u].x);
            d1 += p[u] * bf16_hi(vw[u].x);
            d2 += p[u] * bf16_lo(vw[u].y);
            d3 += p[u] * bf16_hi(vw[u].y);
        }
        o0 = o0 * alpha + d0;
        o1 = o1 * alpha + d1;
        o2 = o2 * alpha + d2;
        o3 = o3 * alpha + d3;
        m = m_new;
    }
    for (; i < i1; ++i) {
        const int64_t row = (key(i) * a.Hkv + j) * 32 + lane;
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
// One CTA per head: thread s weighs split s (2^(m_s - m)), then thread d adds
// the weighted split outputs of dimension d in split order.
__global__ void __launch_bounds__(128) k_dec_combine(DecArgs a, __nv_bfloat16* __restrict__ out)
{
    __shared__ float w_s[kDecSplits];
    __shared__ float red[4];
    const int h = blockIdx.x, d = threadIdx.x;
    const float* ph = a.part + static_cast<int64_t>(h) * a.splits * 130;
    float m = -INFINITY;
    for (int s = threadIdx.x; s < a.splits; s += blockDim.x) m = fmaxf(m, ph[s * 130]);
    m = block_max256(m, red);
    float l = 0.f;
    for (int s = threadIdx.x; s < a.splits; s += blockDim.x) {
        const float ms = ph[s * 130];
        const float w = ms == -INFINITY ? 0.f : exp2f(ms - m);
        w_s[s] = w;
        l += ph[s * 130 + 1] * w;
    }
    l = block_sum256(l, red);  // its barriers also publish w_s
    float o = 0.f;
    for (int s = 0; s < a.splits; ++s) o += ph[s * 130 + 2 + d] * w_s[s];
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
    off = align_up(off + static_cast<size_t>(d.Hq) * ((cap + kDecStat - 1) / kDecStat) * sizeof(float2), kAlign);  // zpart
    off = align_up(off + (kTopkPasses * 256 + (kTopkPasses + 1) * 4) * sizeof(int32_t), kAlign);  // top-k hist, state
    off = align_up(off + static_cast<size_t>(topk_max_chunks(d)) * sizeof(int2), kAlign);          // top-k counts
    return off;
}


int decode_splits() { return kDecSplits; }

cudaError_t launch_decode_step(const Derived& d, int64_t t, const void* q, const void* k, const void* v,
                               uint8_t* cache, void* out, uint8_t* ws, uint64_t timeout_ns, cudaStream_t st)
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
    a.status = reinterpret_cast<int32_t*>(ws + kStatusOffset);
    a.timeout_ns = timeout_ns;
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
    a.zpart = reinterpret_cast<float2*>(
        ws + take(static_cast<size_t>(d.Hq) * ((cap + kDecStat - 1) / kDecStat) * sizeof(float2)));
    int32_t* tk_hist = reinterpret_cast<int32_t*>(ws + take((kTopkPasses * 256 + (kTopkPasses + 1) * 4) * sizeof(int32_t)));
    int2* tk_counts = reinterpret_cast<int2*>(ws + take(static_cast<size_t>(topk_max_chunks(d)) * sizeof(int2)));

    const auto* qb = static_cast<const __nv_bfloat16*>(q);
    k_dec_gate<<<1, 256, 0, st>>>(a, qb);
    const int64_t n_cand = window_start(a, t) - d.n_sink;
    if (n_cand > 0) {
        cudaError_t e0;
        if ((d.g == 1 || d.g == 2 || d.g == 4 || d.g == 8) && d.Hkv <= kDtMaxHkv) {
            // tensor cores, keys streamed by TMA
            const int64_t tiles = (n_cand + 127) / 128;
            a.n_stat = static_cast<int>(tiles);
            CUtensorMap tk;
            if (!scale_host::make_token_major_map(&tk, k, kHeadDim, d.Hkv, d.N, 64, 128)) return cudaErrorInvalidValue;
            int dev = 0, sms = 0;
            e0 = cudaGetDevice(&dev);
            if (e0 == cudaSuccess) e0 = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            if (e0 != cudaSuccess) return e0;
            const int64_t items = tiles * d.Hkv;
            const unsigned grid = static_cast<unsigned>(items < sms ? items : sms);
            auto kern = d.g == 1 ? k_dec_logits_tc<1> : d.g == 2 ? k_dec_logits_tc<2>
                      : d.g == 4 ? k_dec_logits_tc<4> : k_dec_logits_tc<8>;
            e0 = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kDtSmem));
            if (e0 != cudaSuccess) return e0;
            kern<<<grid, kDtThreads, kDtSmem, st>>>(tk, a, qb);
        } else if (d.g == 1 || d.g == 2 || d.g == 4 || d.g == 8) {
            a.n_stat = static_cast<int>((n_cand + kDecStat - 1) / kDecStat);
            auto kern = d.g == 1 ? k_dec_logits<1> : d.g == 2 ? k_dec_logits<2> : d.g == 4 ? k_dec_logits<4>
                                                                                         : k_dec_logits<8>;
            const size_t smem = static_cast<size_t>(d.Hq) * kHeadDim * sizeof(float);
            e0 = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
            if (e0 != cudaSuccess) return e0;
            kern<<<static_cast<unsigned>((n_cand + kDecBlockKeys - 1) / kDecBlockKeys), 256, smem, st>>>(
                a, qb, static_cast<const uint4*>(k));
        } else {
            a.n_stat = static_cast<int>((n_cand + kDecStat - 1) / kDecStat);
            const size_t smem = 2 * static_cast<size_t>(d.Hq) * kHeadDim * sizeof(float);
            e0 = cudaFuncSetAttribute(k_dec_logits_any, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      static_cast<int>(smem));
            if (e0 != cudaSuccess) return e0;
            k_dec_logits_any<<<static_cast<unsigned>((n_cand + 127) / 128), 256, smem, st>>>(
                a, qb, static_cast<const uint4*>(k));
        }
        k_dec_stats<<<d.Hq, 256, 0, st>>>(a, a.n_stat);
        k_dec_vote<<<static_cast<unsigned>((t + 1 + 255) / 256), 256, 0, st>>>(a);
        // top-k of the one-unit table [t, t + 1] kept in the cache, gated on the retrieval flag
        Derived du = d;
        du.L = 1;
        du.B = 1;
        du.nb = d.N;
        const Units ut{a.units, a.units + 2, 0, d.N, 1, static_cast<int>(d.N)};
        const TopkScratch scratch{tk_hist, tk_hist + kTopkPasses * 256, tk_counts, topk_max_chunks(du)};
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
