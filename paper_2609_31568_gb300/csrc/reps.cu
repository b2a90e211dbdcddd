// reps.cu -- step (a) of the SCR prefill path: block representative keys,
// sub-chunk fingerprints (Eq. 6) with their norms (Sec. V-A1), and
// anchor-based clustering (Eq. 8, Algorithm 1) inside each outer chunk.
//
// All four kernels stream their inputs once from HBM with 16-byte loads and
// reduce in a fixed order, so their results are bit-reproducible run to run,
// and each works on a range of outer chunks with the same per-element
// arithmetic as over the whole sequence.
#include <cuda_bf16.h>

#include "scale_internal.h"

namespace scale {
namespace {

__device__ __forceinline__ void add_bf16x8(float (&acc)[8], const uint4 x)
{
    const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        acc[2 * i] += __uint_as_float(w[i] << 16);
        acc[2 * i + 1] += __uint_as_float(w[i] & 0xFFFF0000u);
    }
}

__device__ __forceinline__ uint4 ld_stream(const uint4* p)
{
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

// Representative key of block b for every KV head: the mean of the block's
// keys. One CTA per block, `groups` row groups of row_chunks threads: thread
// c of group g owns elements [8c, 8c+8) of the token rows g, g + groups, ...
// of the block (every row read as one coalesced span), with 8 loads in
// flight; the groups' sums are then added in group order, so the result is
// bit-reproducible. Grid: the blocks [b_base, b_base + gridDim.x).
constexpr int kRepGroups = 4;  // row groups when H_kv * 16 * 4 threads fit a CTA

__global__ void __launch_bounds__(1024) k_block_reps(const uint4* __restrict__ k, KvPaging pg, int64_t N,
                                                      int row_chunks, int groups, int B, int64_t nb,
                                                      int64_t b_base, float* __restrict__ reps)
{
    extern __shared__ float4 part[];  // [groups][row_chunks][2]
    const int c = threadIdx.x % row_chunks;
    const int g = threadIdx.x / row_chunks;
    const int64_t b = b_base + blockIdx.x;
    const int64_t t0 = b * B;
    const int64_t t1 = (t0 + B < N) ? t0 + B : N;
    float acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    const uint4* src = k + c;
    const uint4 zero = make_uint4(0, 0, 0, 0);
    int64_t t = t0 + g;
    for (; t + 7 * groups < t1; t += 8 * groups) {
        uint4 x[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int64_t r = kv_row(pg, t + i * groups);  // -1: a page outside the pool reads as zeros
            x[i] = r < 0 ? zero : ld_stream(src + r * row_chunks);
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) add_bf16x8(acc, x[i]);
    }
    for (; t < t1; t += groups) {
        const int64_t r = kv_row(pg, t);
        add_bf16x8(acc, r < 0 ? zero : ld_stream(src + r * row_chunks));
    }
    part[(g * row_chunks + c) * 2] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    part[(g * row_chunks + c) * 2 + 1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    __syncthreads();
    if (g != 0) return;
    for (int gg = 1; gg < groups; ++gg) {
        const float4 lo = part[(gg * row_chunks + c) * 2], hi = part[(gg * row_chunks + c) * 2 + 1];
        acc[0] += lo.x; acc[1] += lo.y; acc[2] += lo.z; acc[3] += lo.w;
        acc[4] += hi.x; acc[5] += hi.y; acc[6] += hi.z; acc[7] += hi.w;
    }
    // acc held group 0's sum; the groups are added in order for every element
    const float cnt = static_cast<float>(t1 - t0);
    const int j = c / (kHeadDim / 8);
    const int d0 = (c % (kHeadDim / 8)) * 8;
    float4* dst = reinterpret_cast<float4*>(reps + (static_cast<int64_t>(j) * nb + b) * kHeadDim + d0);
    dst[0] = make_float4(acc[0] / cnt, acc[1] / cnt, acc[2] / cnt, acc[3] / cnt);
    dst[1] = make_float4(acc[4] / cnt, acc[5] / cnt, acc[6] / cnt, acc[7] / cnt);
}

// Fingerprint v_i (Eq. 6): the mean of the multi-head queries of sub-chunk i.
// One CTA per (sub-chunk, group of 32 sixteen-byte columns, i.e. 256 of the
// H_q * 128 dimensions). Warp w sums the tokens w, w + 16, w + 32, ... of the
// sub-chunk for its lane's column, so every token row is read as one 512-byte
// span per warp; the 16 warps' sums are then added in warp order, divided by
// |X_i| and written, together with the group's sum of squares (the norm of
// Sec. V-A1 adds those in group order). The order is fixed, so the result is
// bit-reproducible and the same for a sub-chunk whichever range of sub-chunks
// a launch covers. Grid (sub-chunks [m0, m0 + gridDim.x), column groups).
constexpr int kFpWarps = 16;
constexpr int kFpGroupCols = 32;  // 16-byte columns per CTA

__global__ void __launch_bounds__(32 * kFpWarps) k_fingerprint(const uint4* __restrict__ q, int64_t N, int D8,
                                                               int L, int64_t m0, float* __restrict__ fp,
                                                               float* __restrict__ ss_part)
{
    __shared__ float4 red[kFpWarps][kFpGroupCols * 2];
    __shared__ float wsum[8];
    const int64_t i = m0 + blockIdx.x;
    const int cg = blockIdx.y;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int c = cg * kFpGroupCols + lane;
    const int64_t t0 = i * L;
    const int64_t t1 = (t0 + L < N) ? t0 + L : N;
    float acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    if (c < D8) {
        const uint4* src = q + c;
        int64_t t = t0 + w;
        for (; t + 7 * kFpWarps < t1; t += 8 * kFpWarps) {
            uint4 x[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) x[u] = ld_stream(src + (t + u * kFpWarps) * D8);
#pragma unroll
            for (int u = 0; u < 8; ++u) add_bf16x8(acc, x[u]);
        }
        for (; t < t1; t += kFpWarps) add_bf16x8(acc, ld_stream(src + t * D8));
    }
    red[w][2 * lane] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    red[w][2 * lane + 1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    __syncthreads();
    if (threadIdx.x < kFpGroupCols * 8) {
        // thread e owns element e of the group: column e / 8, lane e % 8 of it
        const int e = threadIdx.x;
        const float* flat = reinterpret_cast<const float*>(&red[0][0]);
        float v = 0.f;
        for (int ww = 0; ww < kFpWarps; ++ww) v += flat[ww * kFpGroupCols * 8 + e];
        v = v / static_cast<float>(t1 - t0);
        const int col = cg * kFpGroupCols + e / 8;
        float sq = 0.f;
        if (col < D8) {
            fp[i * static_cast<int64_t>(D8) * 8 + static_cast<int64_t>(col) * 8 + (e & 7)] = v;
            sq = v * v;
        }
        for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xFFFFFFFFu, sq, o);
        if (lane == 0) wsum[w] = sq;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.f;
        for (int ww = 0; ww < kFpGroupCols * 8 / 32; ++ww) t += wsum[ww];
        ss_part[i * gridDim.y + cg] = t;
    }
}

// ||v_i||_2 from the column groups' sums of squares, added in a fixed order
// (lane-strided, then a butterfly that leaves the same value in every lane).
// Warp-collective.
__device__ __forceinline__ float fp_norm(const float* __restrict__ ss_part, int groups, int i)
{
    const int lane = threadIdx.x & 31;
    float s = 0.f;
    for (int g = lane; g < groups; g += 32) s += ss_part[static_cast<int64_t>(i) * groups + g];
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
    return sqrtf(s);
}

// gram[i][d] = cos(v_i, v_{i+d}) = v~_i . v~_{i+d} for 1 <= d < S_max and i+d
// in the same outer chunk; 0 when either norm is 0. One warp per (i, d);
// one CTA per i in [m0, m0 + gridDim.x).
__global__ void k_gram(const float* __restrict__ fp, const float* __restrict__ ss_part, int groups, int D,
                       int M, int S_max, int per_outer, int m0, float* __restrict__ gram)
{
    const int i = m0 + static_cast<int>(blockIdx.x);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nw = blockDim.x >> 5;
    const int chunk_end = min(M, (i / per_outer + 1) * per_outer);
    for (int d = warp + 1; d < S_max; d += nw) {
        const int j = i + d;
        if (j >= chunk_end) continue;
        const float4* a = reinterpret_cast<const float4*>(fp + static_cast<int64_t>(i) * D);
        const float4* b = reinterpret_cast<const float4*>(fp + static_cast<int64_t>(j) * D);
        // 16-byte loads, four independent FMA chains (D is a multiple of 128)
        float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll 8
        for (int c = lane; c < D / 4; c += 32) {
            const float4 x = a[c], y = b[c];
            s0 = fmaf(x.x, y.x, s0);
            s1 = fmaf(x.y, y.y, s1);
            s2 = fmaf(x.z, y.z, s2);
            s3 = fmaf(x.w, y.w, s3);
        }
        float s = (s0 + s1) + (s2 + s3);
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
        const float na = fp_norm(ss_part, groups, i), nb = fp_norm(ss_part, groups, j);  // whole warp
        if (lane == 0) gram[static_cast<int64_t>(i) * S_max + d] = (na > 0.f && nb > 0.f) ? s / (na * nb) : 0.f;
    }
}

// Exclusive block scan of 0/1 flags; returns this thread's exclusive prefix,
// *total receives the block total.
__device__ int block_exclusive_scan(int f, int* sh, int* total)
{
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    int x = f;
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xFFFFFFFFu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) sh[w] = x;
    __syncthreads();
    if (threadIdx.x == 0) {
        int run = 0;
        for (int i = 0; i < nw; ++i) {
            const int t = sh[i];
            sh[i] = run;
            run += t;
        }
        sh[nw] = run;
    }
    __syncthreads();
    const int excl = sh[w] + x - f;
    *total = sh[nw];
    __syncthreads();
    return excl;
}

// Algorithm 1 in the outer chunks [c_begin, c_end) (one thread per chunk walks
// its sub-chunks: the anchor a admits j while cos(v_a, v_j) >= theta and
// |C_a| < S_max), then one block compacts the anchor flags of those chunks
// into unit_start, after the *n_units units of the chunks before c_begin.
__global__ void __launch_bounds__(1024) k_cluster(const float* __restrict__ gram, int M, int S_max,
                                                  int per_outer, float theta, int c_begin, int c_end,
                                                  int32_t* __restrict__ flag,
                                                  int32_t* __restrict__ unit_start,
                                                  int32_t* __restrict__ n_units)
{
    __shared__ int sh[40];
    const bool always = theta <= -1.0f;
    // read before the first barrier; thread 0 rewrites it after the last
    int offset = c_begin == 0 ? 0 : *n_units;
    const int m_begin = c_begin * per_outer;
    const int m_end = min(M, c_end * per_outer);
    for (int c = c_begin + static_cast<int>(threadIdx.x); c < c_end; c += blockDim.x) {
        const int c0 = c * per_outer;
        const int c1 = min(M, c0 + per_outer);
        int a = c0;
        while (a < c1) {
            flag[a] = 1;
            int size = 1, j = a + 1;
            while (j < c1 && size < S_max) {
                const bool admit = always || gram[static_cast<int64_t>(a) * S_max + (j - a)] >= theta;
                if (!admit) break;
                flag[j] = 0;
                ++size;
                ++j;
            }
            a = j;
        }
    }
    __syncthreads();
    for (int base = m_begin; base < m_end; base += blockDim.x) {
        const int i = base + threadIdx.x;
        const int f = (i < m_end) ? flag[i] : 0;
        int total;
        const int excl = block_exclusive_scan(f, sh, &total);
        if (f) unit_start[offset + excl] = i;
        offset += total;
    }
    for (int i = offset + threadIdx.x; i <= M; i += blockDim.x) unit_start[i] = M;
    if (threadIdx.x == 0) *n_units = offset;
}

}  // namespace

int outer_chunks(const Derived& d)
{
    return static_cast<int>((d.M + d.per_outer - 1) / d.per_outer);
}

cudaError_t launch_build_reps_range(const Derived& d, const void* q, const void* k, const KvPaging& pg,
                                    float* reps, float* fingerprints, int32_t* unit_start,
                                    int32_t* n_units, int c_begin, int c_end, uint8_t* ws,
                                    cudaStream_t st)
{
    if (c_begin < 0 || c_end > outer_chunks(d) || c_begin >= c_end) return cudaSuccess;
    const WsLayout lay = ws_layout(d);
    float* ss_part = reinterpret_cast<float*>(ws + lay.fp_ss);
    float* gram = reinterpret_cast<float*>(ws + lay.gram);
    int32_t* flag = reinterpret_cast<int32_t*>(ws + lay.anchor);

    // Tokens [t0, t1) and sub-chunks [m0, m1) of the chunks. A block belongs to
    // the range holding its last token, so every key it averages is present
    // once the chunks up to this range are.
    const int64_t L_outer = static_cast<int64_t>(d.per_outer) * d.L;
    const int64_t t0 = c_begin * L_outer;
    const int64_t t1 = c_end * L_outer < d.N ? c_end * L_outer : d.N;
    const int64_t m0 = static_cast<int64_t>(c_begin) * d.per_outer;
    const int64_t m1 = static_cast<int64_t>(c_end) * d.per_outer < d.M ? static_cast<int64_t>(c_end) * d.per_outer
                                                                         : d.M;
    const int64_t b0 = t0 / d.B;
    const int64_t b1 = t1 == d.N ? d.nb : t1 / d.B;

    const int row_chunks = d.Hkv * (kHeadDim / 8);
    const int groups = row_chunks * kRepGroups <= 1024 ? kRepGroups : 1024 / row_chunks;
    if (reps && b1 > b0)  // block size 1 may skip them: token-level selection reads K itself
        k_block_reps<<<static_cast<unsigned>(b1 - b0), row_chunks * groups,
                       static_cast<size_t>(groups) * row_chunks * 2 * sizeof(float4), st>>>(
            static_cast<const uint4*>(k), pg, d.N, row_chunks, groups, d.B, d.nb, b0, reps);

    const int D8 = d.D / 8;
    const unsigned nm = static_cast<unsigned>(m1 - m0);
    k_fingerprint<<<dim3(nm, d.fp_groups), 32 * kFpWarps, 0, st>>>(static_cast<const uint4*>(q), d.N, D8, d.L,
                                                                   m0, fingerprints, ss_part);
    if (d.S_max > 1) {
        const int warps = d.S_max - 1 < 16 ? d.S_max - 1 : 16;
        k_gram<<<nm, 32 * warps, 0, st>>>(fingerprints, ss_part, d.fp_groups, d.D, static_cast<int>(d.M),
                                          d.S_max, d.per_outer, static_cast<int>(m0), gram);
    }
    k_cluster<<<1, 1024, 0, st>>>(gram, static_cast<int>(d.M), d.S_max, d.per_outer, d.theta, c_begin,
                                  c_end, flag, unit_start, n_units);
    return cudaGetLastError();
}

cudaError_t launch_build_reps(const Derived& d, const void* q, const void* k, const KvPaging& pg,
                              float* reps, float* fingerprints, int32_t* unit_start, int32_t* n_units,
                              uint8_t* ws, cudaStream_t st)
{
    return launch_build_reps_range(d, q, k, pg, reps, fingerprints, unit_start, n_units, 0,
                                   outer_chunks(d), ws, st);
}

}  // namespace scale
