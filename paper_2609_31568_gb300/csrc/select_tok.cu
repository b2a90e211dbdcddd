// select_tok.cu -- token-level selection (block size 1): the selection rule of
// Sec. V-A3 ("Selection function instantiation") applied to every key on its
// own, as the paper does, instead of to block representatives.
//
// For unit u with anchor a(u) and candidate tokens n_sink <= t < W_u,
// W_u = max(0, s_u - n_local) (Eq. 9):
//   z[u][h][t]  = sigma * v_a^(h) . k_t^(h/g)
//   p[u][h][t]  = exp(z - max_t z) / sum_t exp(z - max_t z)     (per head)
//   score[u][t] = sum_h p[u][h][t]                              (soft vote)
// followed by the top-k of select.cu (ties to the lower token, ascending).
//
// The contraction runs on the tensor cores (tcgen05.mma kind::f16, fp32
// accumulation in TMEM) straight from the bf16 keys. The fp32 fingerprint is
// split into three bf16 parts v1 + v2 + v3 that hold it exactly, so the three
// MMAs v_i . k (products of two bf16 values are exact in fp32) sum to the fp32
// dot product up to accumulation order.
//
//   k_tok_split     v_a(u)^(h) -> bf16 parts [3][H_kv][units][g][128]
//   k_tok_score<0>  rows (unit, head) x 128-token columns: per token range,
//                   each row's running max and sum of 2^(z' - m), z' = z log2 e
//   k_tok_merge     per (unit, head): the ranges' (max, sum) merged in order
//   k_tok_score<1>  rows = tokens x columns (unit, head): 2^(z' - m) / sum,
//                   summed over the heads of each unit in a fixed order and
//                   accumulated over the KV heads in shared memory; the CTA
//                   owns its (unit, token) cells, so no atomics are needed.
//
// Each CTA owns a tile of 128 / g units and a range of 128 g tokens (<= 1024).
// Calls of at most 16 units (every call of the Algorithm 2 loop) use
// k_tok_score_s instead: 16 (unit, head) columns per tile, tokens as the MMA
// rows and the three parts side by side in one N = 48 operand.
// Warp 0 lane 0 issues TMA loads (the fingerprint parts of one KV head, then
// 128-token key tiles into a 2-stage ring), warp 1 lane 0 issues the MMAs
// (TMEM: two 128-column accumulators), warps 2-5 run the epilogue. Every wait
// is bounded; on expiry the kernel records SCALE_ERR_TIMEOUT and drains.
#include <cuda_bf16.h>

#include "ptx_sm103.cuh"
#include "scale_internal.h"
#include "tma_host.h"

namespace scale {
namespace {

using namespace scale_ptx;

constexpr int kTokThreads = 192;
constexpr uint32_t kTile = 128 * 128 * 2;   // 128 rows x 128 bf16
constexpr uint32_t kHalfT = kTile / 2;      // one 64-column half
constexpr uint32_t kOffF = 0;               // 3 fingerprint parts
constexpr uint32_t kOffK = 3 * kTile;       // 2 key stages
constexpr uint32_t kOffVote = 5 * kTile;    // pass 1: [units][range] fp32 (64 KB)
constexpr uint32_t kVoteBytes = 64 * 1024;
constexpr uint32_t kSmemTok0 = kOffVote + 1024;
constexpr uint32_t kSmemTok1 = kOffVote + kVoteBytes + 1024;
static_assert(kSmemTok1 <= 227 * 1024 - 2048, "token scoring shared memory");

struct TokArgs {
    Units ut;
    int sc_begin, sc_end;
    int Hq, Hkv, g, U;  // U = units per tile = 128 / g
    int range;          // tokens per CTA (128 g, at most 1024)
    int n_ranges;
    int N, n_sink, n_local;
    int head_split;     // k_tok_score_s pass 0: one KV head per CTA (grid z)
    float scale2;       // sigma * log2(e)
    float2* part;       // [M][H_q][n_ranges] (max, sum) in log2 units
    const float2* stats;  // [M][H_q] (max, 1 / sum)
    float* scores;      // [M][N]
    int32_t* status;
    uint64_t timeout_ns;
    KvPaging pg;
};

struct TokBars {
    uint64_t f_full, f_empty;
    uint64_t k_full[2], k_empty[2];
    uint64_t d_full[2], d_empty[2];
    uint64_t drain;
};

__device__ __forceinline__ void tok_fail(volatile int* abort_flag, int32_t* status)
{
    *abort_flag = 1;
    record_status(status, SCALE_ERR_TIMEOUT);
}

__device__ __forceinline__ int64_t window_start(const TokArgs& a, int u)
{
    int anc;
    int64_t s, e;
    unit_range(a.ut, u, &anc, &s, &e);
    return s - a.n_local > 0 ? s - a.n_local : 0;
}

template <int PASS, int G>
__global__ void __launch_bounds__(kTokThreads, 1)
k_tok_score(const __grid_constant__ CUtensorMap tf, const __grid_constant__ CUtensorMap tk, const TokArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ TokBars bars;
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    __shared__ int s_W[128];
    __shared__ float2 s_col[128];

    const int u_first = unit_lower_bound(a.ut, a.sc_begin);
    const int u_end = unit_lower_bound(a.ut, a.sc_end);
    const int u0 = u_first + static_cast<int>(blockIdx.y) * a.U;
    if (u0 >= u_end) return;
    const int n_u = (u_end - u0 < a.U) ? u_end - u0 : a.U;
    const int x = blockIdx.x;
    const int r0 = x * a.range;
    const int r1 = (r0 + a.range < a.N) ? r0 + a.range : a.N;
    // Candidates of the tile's units end at the last unit's window start.
    const int64_t w_max = window_start(a, u0 + n_u - 1);
    const int c_hi = static_cast<int>(w_max < r1 ? w_max : r1);
    const bool work = c_hi > r0 && c_hi > a.n_sink;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (!work) {
        if (PASS == 1) {  // no candidate in the range: every score is NaN
            for (int ul = 0; ul < n_u; ++ul)
                for (int t = r0 + tid; t < r1; t += blockDim.x)
                    a.scores[static_cast<int64_t>(u0 + ul) * a.N + t] = __int_as_float(0x7FC00000);
        }
        return;
    }
    const int n_tiles = (c_hi - r0 + 127) / 128;

    uint8_t* smem = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
    float* vote = reinterpret_cast<float*>(smem + kOffVote);

    if (tid < 128) s_W[tid] = (tid < n_u) ? static_cast<int>(window_start(a, u0 + tid)) : 0;
    if (tid == 0) {
        abort_flag = 0;
        mbar_init(&bars.f_full, 1);
        mbar_init(&bars.f_empty, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars.k_full[i], 1);
            mbar_init(&bars.k_empty[i], 1);
            mbar_init(&bars.d_full[i], 1);
            mbar_init(&bars.d_empty[i], 128);
        }
        mbar_init(&bars.drain, 1);
        fence_barrier_init();
    }
    if (PASS == 1)
        for (int i = tid; i < a.U * a.range; i += blockDim.x) vote[i] = 0.f;
    if (warp == 1) {
        tmem_alloc(&tmem_slot, 256);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&tf);
            tma_prefetch_desc(&tk);
            int gt = 0;
            int issued_k0 = 0, issued_k1 = 0, issued_f = 0;
            for (int j = 0; j < a.Hkv && !abort_flag; ++j) {
                if (j > 0 && !mbar_wait_bounded(&bars.f_empty, (j - 1) & 1, a.timeout_ns, &abort_flag)) {
                    tok_fail(&abort_flag, a.status);
                    break;
                }
                mbar_arrive_expect_tx(&bars.f_full, 3 * kTile);
                ++issued_f;
                for (int s = 0; s < 3; ++s)
                    for (int hf = 0; hf < 2; ++hf)
                        tma_load_4d(smem + kOffF + s * kTile + hf * kHalfT, &tf, &bars.f_full, hf * 64,
                                    u0 * G, j, s);
                for (int i = 0; i < n_tiles; ++i, ++gt) {
                    const int st = gt & 1;
                    if (gt >= 2 && !mbar_wait_bounded(&bars.k_empty[st], ((gt >> 1) - 1) & 1, a.timeout_ns, &abort_flag)) {
                        tok_fail(&abort_flag, a.status);
                        break;
                    }
                    mbar_arrive_expect_tx(&bars.k_full[st], kTile);
                    if (st) ++issued_k1; else ++issued_k0;
                    // two 64-row boxes per half: each lies inside one KV page
                    const int32_t ra = kv_row_tma(a.pg, r0 + 128 * i);
                    const int32_t rb = kv_row_tma(a.pg, r0 + 128 * i + 64);
                    for (int hf = 0; hf < 2; ++hf) {
                        uint8_t* dst = smem + kOffK + st * kTile + hf * kHalfT;
                        tma_load_3d(dst, &tk, &bars.k_full[st], hf * 64, j, ra);
                        tma_load_3d(dst + kHalfT / 2, &tk, &bars.k_full[st], hf * 64, j, rb);
                    }
                }
            }
            if (abort_flag) {
                if (issued_f) mbar_wait_bounded(&bars.f_full, (issued_f - 1) & 1, a.timeout_ns, nullptr);
                if (issued_k0) mbar_wait_bounded(&bars.k_full[0], (issued_k0 - 1) & 1, a.timeout_ns, nullptr);
                if (issued_k1) mbar_wait_bounded(&bars.k_full[1], (issued_k1 - 1) & 1, a.timeout_ns, nullptr);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, 128, 0);
            const uint64_t fdesc0 = sdesc_sw128(smem_addr(smem + kOffF), 16, 1024);
            const uint64_t kdesc0 = sdesc_sw128(smem_addr(smem + kOffK), 16, 1024);
            constexpr uint64_t kStep = kTile >> 4;
            bool ok = true;
            int gt = 0;
            for (int j = 0; ok && j < a.Hkv; ++j) {
                if (!mbar_wait_bounded(&bars.f_full, j & 1, a.timeout_ns, &abort_flag)) { ok = false; break; }
                for (int i = 0; i < n_tiles; ++i, ++gt) {
                    const int st = gt & 1;
                    if (!mbar_wait_bounded(&bars.k_full[st], (gt >> 1) & 1, a.timeout_ns, &abort_flag)) { ok = false; break; }
                    if (gt >= 2 && !mbar_wait_bounded(&bars.d_empty[st], ((gt >> 1) - 1) & 1, a.timeout_ns, &abort_flag)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t d = tmem + st * 128;
                    const uint64_t kd = kdesc0 + st * kStep;
#pragma unroll
                    for (int s = 0; s < 3; ++s) {
                        const uint64_t fd = fdesc0 + s * kStep;
                        if (PASS == 0)
                            mma_ss_k128<kHalfT>(d, fd, kd, idesc, s > 0 ? 1u : 0u);
                        else
                            mma_ss_k128<kHalfT>(d, kd, fd, idesc, s > 0 ? 1u : 0u);
                    }
                    mma_commit(&bars.d_full[st]);
                    mma_commit(&bars.k_empty[st]);
                }
                if (ok) mma_commit(&bars.f_empty);
            }
            if (!ok) {
                tok_fail(&abort_flag, a.status);
                mma_commit(&bars.drain);
                mbar_wait_bounded(&bars.drain, 0, a.timeout_ns, nullptr);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int q = warp & 3;  // TMEM lane quarter this warp may access
        const int r = q * 32 + lane;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(q * 32) << 16);
        bool ok = true;
        int gt = 0;
        if (PASS == 0) {
            const int ul = r / G, hl = r % G;
            const bool valid = ul < n_u;
            const int lo = a.n_sink, hi = valid ? (s_W[ul] < r1 ? s_W[ul] : r1) : 0;
            for (int j = 0; j < a.Hkv; ++j) {
                float m = -INFINITY, sum = 0.f;
                for (int i = 0; i < n_tiles; ++i, ++gt) {
                    const int st = gt & 1;
                    if (!ok) continue;
                    const bool got = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(&bars.d_full[st], (gt >> 1) & 1, a.timeout_ns, &abort_flag));
                    if (!got) { ok = false; continue; }
                    tc_fence_after();
                    uint32_t zr[128];
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        tmem_ld32(lane_base + st * 128 + c * 32, *reinterpret_cast<uint32_t(*)[32]>(&zr[c * 32]));
                    tmem_ld_wait();
                    tc_fence_before();
                    mbar_arrive(&bars.d_empty[st]);
                    const int t0 = r0 + 128 * i;
                    if (t0 + 127 < lo || t0 >= hi) continue;  // no candidate of this row here
                    float* z = reinterpret_cast<float*>(zr);
                    float tmax = -INFINITY;
#pragma unroll
                    for (int c = 0; c < 128; ++c) {
                        const int t = t0 + c;
                        z[c] = (t >= lo && t < hi) ? z[c] * a.scale2 : -INFINITY;
                        tmax = fmaxf(tmax, z[c]);
                    }
                    const float m_new = fmaxf(m, tmax);
                    float acc = 0.f;
#pragma unroll
                    for (int c = 0; c < 128; ++c) acc += ex2(z[c] - m_new);
                    sum = sum * ex2(m - m_new) + acc;
                    m = m_new;
                }
                if (ok && valid)
                    a.part[(static_cast<int64_t>(u0 + ul) * a.Hq + j * G + hl) * a.n_ranges + x] = make_float2(m, sum);
            }
        } else {
            // Every epilogue warp runs the same sequence of named barriers,
            // also after a failed wait (it then skips the work).
            for (int j = 0; j < a.Hkv; ++j) {
                // column statistics of this KV head's (unit, head) columns
                named_barrier(1, 128);
                {
                    const int ul = r / G, hl = r % G;
                    s_col[r] = (ul < n_u) ? a.stats[static_cast<int64_t>(u0 + ul) * a.Hq + j * G + hl]
                                          : make_float2(0.f, 0.f);
                }
                named_barrier(1, 128);
                for (int i = 0; i < n_tiles; ++i, ++gt) {
                    const int st = gt & 1;
                    if (!ok) continue;
                    const bool got = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(&bars.d_full[st], (gt >> 1) & 1, a.timeout_ns, &abort_flag));
                    if (!got) { ok = false; continue; }
                    tc_fence_after();
                    uint32_t zr[128];
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        tmem_ld32(lane_base + st * 128 + c * 32, *reinterpret_cast<uint32_t(*)[32]>(&zr[c * 32]));
                    tmem_ld_wait();
                    tc_fence_before();
                    mbar_arrive(&bars.d_empty[st]);
                    const float* z = reinterpret_cast<const float*>(zr);
                    const int t = r0 + 128 * i + r;
                    if (t < a.n_sink || t >= c_hi) continue;
                    float* vrow = vote + 128 * i + r;
#pragma unroll
                    for (int ul = 0; ul < 128 / G; ++ul) {
                        float acc = 0.f;
#pragma unroll
                        for (int hl = 0; hl < G; ++hl) {
                            const int c = ul * G + hl;
                            const float2 cs = s_col[c];
                            acc += ex2(z[c] * a.scale2 - cs.x) * cs.y;
                        }
                        if (ul < n_u && t < s_W[ul]) vrow[ul * a.range] += acc;
                    }
                }
            }
            bool all_ok = __all_sync(0xFFFFFFFFu, ok && !abort_flag);
            named_barrier(1, 128);
            if (all_ok) {
                for (int ul = 0; ul < n_u; ++ul) {
                    float* dst = a.scores + static_cast<int64_t>(u0 + ul) * a.N;
                    for (int tt = r; tt < r1 - r0; tt += 128) {
                        const int t = r0 + tt;
                        dst[t] = (t >= a.n_sink && t < s_W[ul]) ? vote[ul * a.range + tt]
                                                                 : __int_as_float(0x7FC00000);
                    }
                }
            }
            ok = all_ok;
        }
        if (!ok) tok_fail(&abort_flag, a.status);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 256);
    }
}

// ---- the same two passes for calls with few units (every call of the
// Algorithm 2 loop covers one cluster or one sub-chunk): a unit tile of
// 16 / G units, i.e. 16 (unit, head) columns. The 128 tokens of a key tile
// are the MMA rows and the three bf16 parts of the 16 fingerprint columns sit
// side by side in one N = 48 operand (part s at columns [16 s, 16 s + 16)),
// so one MMA per K-step yields the three partial dot products: 8 MMAs per key
// tile instead of 24, and a 12 KB fingerprint tile per KV head instead of
// 96 KB. Pass 0 keeps a running (max, sum) per column in each token's thread
// and merges the 128 threads once per KV head (a fixed shuffle tree, then
// the four warps in order); pass 1 keeps each token's votes in registers.
// For parallelism when the sequence has few token ranges, pass 0 then runs
// one CTA per KV head (grid z; its partials are per (unit, head) anyway) and
// pass 1 (NARROW) one CTA per 128 tokens (the votes are per token); with many
// ranges the CTAs keep all KV heads and whole ranges, which amortises the
// fingerprint loads and the pipeline start over more key tiles.
constexpr int kNc = 16;                        // (unit, head) columns of a small tile
constexpr int kRange1 = 128;                   // narrow pass 1: tokens per CTA
constexpr int kFewRanges = 1024;               // below this many ranges: the split grids
constexpr uint32_t kFsHalf = 3 * kNc * 128;    // one 64-column half of the 48-row operand: 6 KB
constexpr uint32_t kOffFs = 0;                 // fingerprint parts, 12 KB
constexpr uint32_t kOffKs = 2 * kFsHalf;       // 2 key stages (a multiple of 1024)
constexpr uint32_t kSmemTokS = kOffKs + 2 * kTile + 1024;
static_assert(kOffKs % 1024 == 0, "key stages must stay 1024-aligned");

// (m, s) of a sum of 2^(z - m) terms merged with another: both in log2 units.
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2)
{
    const float mn = fmaxf(m, m2);
    if (mn == -INFINITY) return;
    s = s * ex2(m - mn) + s2 * ex2(m2 - mn);
    m = mn;
}

template <int PASS, int G, bool NARROW>
__global__ void __launch_bounds__(kTokThreads, 2)
k_tok_score_s(const __grid_constant__ CUtensorMap tfs, const __grid_constant__ CUtensorMap tk, const TokArgs a)
{
    constexpr int US = kNc / G;  // units of the tile
    extern __shared__ uint8_t smem_raw[];
    __shared__ TokBars bars;
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    __shared__ int s_W[US];
    __shared__ float2 s_col[kNc];
    __shared__ float2 s_red[4][kNc];

    const int u_first = unit_lower_bound(a.ut, a.sc_begin);
    const int u_end = unit_lower_bound(a.ut, a.sc_end);
    const int u0 = u_first + static_cast<int>(blockIdx.y) * US;
    if (u0 >= u_end) return;
    const int n_u = (u_end - u0 < US) ? u_end - u0 : US;
    const int x = blockIdx.x;
    const int rlen = (PASS == 1 && NARROW) ? kRange1 : a.range;
    const int r0 = x * rlen;
    const int r1 = (r0 + rlen < a.N) ? r0 + rlen : a.N;
    const bool split = PASS == 0 && a.head_split;  // KV heads of this CTA
    const int j_lo = split ? static_cast<int>(blockIdx.z) : 0;
    const int j_hi = split ? j_lo + 1 : a.Hkv;
    const int64_t w_max = window_start(a, u0 + n_u - 1);
    const int c_hi = static_cast<int>(w_max < r1 ? w_max : r1);
    const bool work = c_hi > r0 && c_hi > a.n_sink;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (!work) {
        if (PASS == 1) {  // no candidate in the range: every score is NaN
            for (int ul = 0; ul < n_u; ++ul)
                for (int t = r0 + tid; t < r1; t += blockDim.x)
                    a.scores[static_cast<int64_t>(u0 + ul) * a.N + t] = __int_as_float(0x7FC00000);
        }
        return;
    }
    const int n_tiles = (c_hi - r0 + 127) / 128;

    uint8_t* smem = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
    if (tid < US) s_W[tid] = (tid < n_u) ? static_cast<int>(window_start(a, u0 + tid)) : 0;
    if (tid == 0) {
        abort_flag = 0;
        mbar_init(&bars.f_full, 1);
        mbar_init(&bars.f_empty, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars.k_full[i], 1);
            mbar_init(&bars.k_empty[i], 1);
            mbar_init(&bars.d_full[i], 1);
            mbar_init(&bars.d_empty[i], 128);
        }
        mbar_init(&bars.drain, 1);
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

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&tfs);
            tma_prefetch_desc(&tk);
            int gt = 0;
            int issued_k0 = 0, issued_k1 = 0, issued_f = 0;
            for (int j = j_lo; j < j_hi && !abort_flag; ++j) {
                if (j > j_lo && !mbar_wait_bounded(&bars.f_empty, (j - j_lo - 1) & 1, a.timeout_ns, &abort_flag)) {
                    tok_fail(&abort_flag, a.status);
                    break;
                }
                mbar_arrive_expect_tx(&bars.f_full, 2 * kFsHalf);
                ++issued_f;
                for (int sp = 0; sp < 3; ++sp)
                    for (int hf = 0; hf < 2; ++hf)
                        tma_load_4d(smem + kOffFs + hf * kFsHalf + sp * kNc * 128, &tfs, &bars.f_full, hf * 64,
                                    u0 * G, j, sp);
                for (int i = 0; i < n_tiles; ++i, ++gt) {
                    const int st = gt & 1;
                    if (gt >= 2 && !mbar_wait_bounded(&bars.k_empty[st], ((gt >> 1) - 1) & 1, a.timeout_ns, &abort_flag)) {
                        tok_fail(&abort_flag, a.status);
                        break;
                    }
                    mbar_arrive_expect_tx(&bars.k_full[st], kTile);
                    if (st) ++issued_k1; else ++issued_k0;
                    const int32_t ra = kv_row_tma(a.pg, r0 + 128 * i);
                    const int32_t rb = kv_row_tma(a.pg, r0 + 128 * i + 64);
                    for (int hf = 0; hf < 2; ++hf) {
                        uint8_t* dst = smem + kOffKs + st * kTile + hf * kHalfT;
                        tma_load_3d(dst, &tk, &bars.k_full[st], hf * 64, j, ra);
                        tma_load_3d(dst + kHalfT / 2, &tk, &bars.k_full[st], hf * 64, j, rb);
                    }
                }
            }
            if (abort_flag) {
                if (issued_f) mbar_wait_bounded(&bars.f_full, (issued_f - 1) & 1, a.timeout_ns, nullptr);
                if (issued_k0) mbar_wait_bounded(&bars.k_full[0], (issued_k0 - 1) & 1, a.timeout_ns, nullptr);
                if (issued_k1) mbar_wait_bounded(&bars.k_full[1], (issued_k1 - 1) & 1, a.timeout_ns, nullptr);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, 3 * kNc, 0);
            const uint64_t fdesc = sdesc_sw128(smem_addr(smem + kOffFs), 16, 1024);
            const uint64_t kdesc0 = sdesc_sw128(smem_addr(smem + kOffKs), 16, 1024);
            constexpr uint64_t kStep = kTile >> 4;
            bool ok = true;
            int gt = 0;
            for (int j = j_lo; ok && j < j_hi; ++j) {
                if (!mbar_wait_bounded(&bars.f_full, (j - j_lo) & 1, a.timeout_ns, &abort_flag)) { ok = false; break; }
                for (int i = 0; i < n_tiles; ++i, ++gt) {
                    const int st = gt & 1;
                    if (!mbar_wait_bounded(&bars.k_full[st], (gt >> 1) & 1, a.timeout_ns, &abort_flag)) { ok = false; break; }
                    if (gt >= 2 && !mbar_wait_bounded(&bars.d_empty[st], ((gt >> 1) - 1) & 1, a.timeout_ns, &abort_flag)) { ok = false; break; }
                    tc_fence_after();
                    // rows: the tile's 128 tokens (A = keys), columns: 3 parts x 16
                    mma_ss_k128_ab<kHalfT, kFsHalf>(tmem + st * 64, kdesc0 + st * kStep, fdesc, idesc, 0u);
                    mma_commit(&bars.d_full[st]);
                    mma_commit(&bars.k_empty[st]);
                }
                if (ok) mma_commit(&bars.f_empty);
            }
            if (!ok) {
                tok_fail(&abort_flag, a.status);
                mma_commit(&bars.drain);
                mbar_wait_bounded(&bars.drain, 0, a.timeout_ns, nullptr);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int q = warp & 3;  // TMEM lane quarter this warp may access
        const int r = q * 32 + lane;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(q * 32) << 16);
        bool ok = true;
        int gt = 0;
        // z of this thread's token for the 16 columns: the three parts added
        auto load_z = [&](int st, float (&z)[kNc]) {
            uint32_t p0[16], p1[16], p2[16];
            tmem_ld16(lane_base + st * 64, p0);
            tmem_ld16(lane_base + st * 64 + kNc, p1);
            tmem_ld16(lane_base + st * 64 + 2 * kNc, p2);
            tmem_ld_wait();
#pragma unroll
            for (int c = 0; c < kNc; ++c)
                z[c] = (__uint_as_float(p0[c]) + __uint_as_float(p1[c])) + __uint_as_float(p2[c]);
        };
        if (PASS == 0) {
            for (int j = j_lo; j < j_hi; ++j) {
                float m[kNc], sm[kNc];
#pragma unroll
                for (int c = 0; c < kNc; ++c) {
                    m[c] = -INFINITY;
                    sm[c] = 0.f;
                }
                for (int i = 0; i < n_tiles; ++i, ++gt) {
                    const int st = gt & 1;
                    if (!ok) continue;
                    const bool got = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(&bars.d_full[st], (gt >> 1) & 1, a.timeout_ns, &abort_flag));
                    if (!got) { ok = false; continue; }
                    tc_fence_after();
                    float z[kNc];
                    load_z(st, z);
                    tc_fence_before();
                    mbar_arrive(&bars.d_empty[st]);
                    const int t = r0 + 128 * i + r;
                    if (t < a.n_sink || t >= c_hi) continue;
#pragma unroll
                    for (int c = 0; c < kNc; ++c) {
                        const int ul = c / G;
                        if (ul < n_u && t < s_W[ul]) {
                            const float zz = z[c] * a.scale2;
                            const float mn = fmaxf(m[c], zz);
                            sm[c] = sm[c] * ex2(m[c] - mn) + ex2(zz - mn);
                            m[c] = mn;
                        }
                    }
                }
                // merge the 128 tokens' (max, sum) per column: lanes, then warps in order
#pragma unroll
                for (int c = 0; c < kNc; ++c)
                    for (int o = 16; o > 0; o >>= 1) {
                        const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m[c], o);
                        const float s2 = __shfl_xor_sync(0xFFFFFFFFu, sm[c], o);
                        lse_merge(m[c], sm[c], m2, s2);
                    }
                if (lane < kNc) {
                    float mv = m[0], sv = sm[0];
#pragma unroll
                    for (int c = 1; c < kNc; ++c)
                        if (lane == c) {
                            mv = m[c];
                            sv = sm[c];
                        }
                    s_red[q][lane] = make_float2(mv, sv);
                }
                named_barrier(1, 128);
                if (r < kNc && ok) {
                    const int ul = r / G, hl = r % G;
                    float mv = s_red[0][r].x, sv = s_red[0][r].y;
                    for (int w = 1; w < 4; ++w) lse_merge(mv, sv, s_red[w][r].x, s_red[w][r].y);
                    if (ul < n_u)
                        a.part[(static_cast<int64_t>(u0 + ul) * a.Hq + j * G + hl) * a.n_ranges + x] =
                            make_float2(mv, sv);
                }
                named_barrier(1, 128);
            }
        } else {
            // votes of this thread's token in each key tile of the range, per unit
            constexpr int kTiles = NARROW ? kRange1 / 128 : (G < 8 ? G : 8);  // the range's key tiles
            float vote[kTiles][US];
#pragma unroll
            for (int i = 0; i < kTiles; ++i)
#pragma unroll
                for (int ul = 0; ul < US; ++ul) vote[i][ul] = 0.f;
            for (int j = 0; j < a.Hkv; ++j) {
                named_barrier(1, 128);
                if (r < kNc) {
                    const int ul = r / G, hl = r % G;
                    s_col[r] = (ul < n_u) ? a.stats[static_cast<int64_t>(u0 + ul) * a.Hq + j * G + hl]
                                          : make_float2(0.f, 0.f);
                }
                named_barrier(1, 128);
#pragma unroll
                for (int i = 0; i < kTiles; ++i) {
                    if (i >= n_tiles) continue;
                    const int st = gt & 1;
                    const int ph = (gt >> 1) & 1;
                    ++gt;
                    if (!ok) continue;
                    const bool got = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(&bars.d_full[st], ph, a.timeout_ns, &abort_flag));
                    if (!got) { ok = false; continue; }
                    tc_fence_after();
                    float z[kNc];
                    load_z(st, z);
                    tc_fence_before();
                    mbar_arrive(&bars.d_empty[st]);
                    const int t = r0 + 128 * i + r;
                    if (t < a.n_sink || t >= c_hi) continue;
#pragma unroll
                    for (int ul = 0; ul < US; ++ul) {
                        float acc = 0.f;
#pragma unroll
                        for (int hl = 0; hl < G; ++hl) {
                            const int c = ul * G + hl;
                            const float2 cs = s_col[c];
                            acc += ex2(z[c] * a.scale2 - cs.x) * cs.y;
                        }
                        if (ul < n_u && t < s_W[ul]) vote[i][ul] += acc;
                    }
                }
            }
            if (__all_sync(0xFFFFFFFFu, ok && !abort_flag)) {
#pragma unroll
                for (int i = 0; i < kTiles; ++i) {
                    const int t = r0 + 128 * i + r;
                    if (t >= r1) continue;
#pragma unroll
                    for (int ul = 0; ul < US; ++ul)
                        if (ul < n_u)
                            a.scores[static_cast<int64_t>(u0 + ul) * a.N + t] =
                                (t >= a.n_sink && t < s_W[ul]) ? vote[i][ul] : __int_as_float(0x7FC00000);
                }
            } else {
                ok = false;
            }
        }
        if (!ok) tok_fail(&abort_flag, a.status);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 128);
    }
}

// v_a(u)^(h) (fp32) -> three bf16 parts; row (u, h) of KV head j = h / g at
// [part][j][u][h % g][128].
__global__ void __launch_bounds__(128) k_tok_split(TokArgs a, const float* __restrict__ fp,
                                                   __nv_bfloat16* __restrict__ parts, int M)
{
    const int u_first = unit_lower_bound(a.ut, a.sc_begin);
    const int u_end = unit_lower_bound(a.ut, a.sc_end);
    const int u = u_first + static_cast<int>(blockIdx.x) / a.Hq;
    const int h = static_cast<int>(blockIdx.x) % a.Hq;
    if (u >= u_end) return;
    int anc;
    int64_t s, e;
    unit_range(a.ut, u, &anc, &s, &e);
    const int d = threadIdx.x;
    const float v = fp[static_cast<int64_t>(anc) * a.Hq * kHeadDim + h * kHeadDim + d];
    const __nv_bfloat16 v1 = __float2bfloat16_rn(v);
    const float r1 = v - __bfloat162float(v1);
    const __nv_bfloat16 v2 = __float2bfloat16_rn(r1);
    const __nv_bfloat16 v3 = __float2bfloat16_rn(r1 - __bfloat162float(v2));
    const int j = h / a.g, hl = h % a.g;
    const int64_t plane = static_cast<int64_t>(a.Hkv) * M * a.g * kHeadDim;
    const int64_t off = ((static_cast<int64_t>(j) * M + u) * a.g + hl) * kHeadDim + d;
    parts[off] = v1;
    parts[plane + off] = v2;
    parts[2 * plane + off] = v3;
}

// One warp per (unit, head): merge the token ranges' (max, sum); the lanes
// take ranges in a fixed interleave and combine in a fixed tree, so the result
// does not depend on scheduling.
__global__ void __launch_bounds__(256) k_tok_merge(TokArgs a)
{
    const int u_first = unit_lower_bound(a.ut, a.sc_begin);
    const int u_end = unit_lower_bound(a.ut, a.sc_end);
    const int64_t i = static_cast<int64_t>(blockIdx.x) * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    const int u = u_first + static_cast<int>(i / a.Hq);
    const int h = static_cast<int>(i % a.Hq);
    if (u >= u_end) return;
    const int64_t W = window_start(a, u);
    const int hi = static_cast<int>(W < a.N ? W : a.N);
    float m = -INFINITY, sum = 0.f;
    if (hi > a.n_sink) {
        const float2* pr = a.part + (static_cast<int64_t>(u) * a.Hq + h) * a.n_ranges;
        const int x0 = a.n_sink / a.range, x1 = (hi + a.range - 1) / a.range;
        for (int xx = x0 + lane; xx < x1; xx += 32) m = fmaxf(m, pr[xx].x);
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
        for (int xx = x0 + lane; xx < x1; xx += 32)
            if (pr[xx].x > -INFINITY) sum += pr[xx].y * ex2(pr[xx].x - m);
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
    }
    if (lane == 0)
        const_cast<float2*>(a.stats)[static_cast<int64_t>(u) * a.Hq + h] =
            make_float2(m, sum > 0.f ? 1.0f / sum : 0.f);
}

template <int G>
cudaError_t run_tok_passes(dim3 grid, int64_t rows, const CUtensorMap& tf, const CUtensorMap& tk,
                           const TokArgs& a, cudaStream_t st)
{
    // set on every launch: the attribute belongs to the current device
    cudaError_t e = cudaFuncSetAttribute(k_tok_score<0, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kSmemTok0));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_tok_score<1, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kSmemTok1));
    if (e != cudaSuccess) return e;
    k_tok_score<0, G><<<grid, kTokThreads, kSmemTok0, st>>>(tf, tk, a);
    k_tok_merge<<<static_cast<unsigned>((rows + 7) / 8), 256, 0, st>>>(a);
    k_tok_score<1, G><<<grid, kTokThreads, kSmemTok1, st>>>(tf, tk, a);
    return cudaGetLastError();
}

// The two passes with small unit tiles (k_tok_score_s): calls of at most
// kSmallUnits units.
constexpr int kSmallUnits = 16;

template <int G, bool NARROW>
cudaError_t run_tok_passes_s(dim3 grid0, dim3 grid1, int64_t rows, const CUtensorMap& tfs,
                             const CUtensorMap& tk, const TokArgs& a, cudaStream_t st)
{
    cudaError_t e = cudaFuncSetAttribute(k_tok_score_s<0, G, NARROW>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kSmemTokS));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_tok_score_s<1, G, NARROW>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kSmemTokS));
    if (e != cudaSuccess) return e;
    k_tok_score_s<0, G, NARROW><<<grid0, kTokThreads, kSmemTokS, st>>>(tfs, tk, a);
    k_tok_merge<<<static_cast<unsigned>((rows + 7) / 8), 256, 0, st>>>(a);
    k_tok_score_s<1, G, NARROW><<<grid1, kTokThreads, kSmemTokS, st>>>(tfs, tk, a);
    return cudaGetLastError();
}

template <int G>
cudaError_t run_tok_passes_s(const Derived& d, int tiles, int64_t rows, const CUtensorMap& tfs,
                             const CUtensorMap& tk, TokArgs a, cudaStream_t st)
{
    const unsigned nt = static_cast<unsigned>(tiles);
    if (a.n_ranges < kFewRanges) {
        a.head_split = 1;
        return run_tok_passes_s<G, true>(dim3(static_cast<unsigned>(a.n_ranges), nt, static_cast<unsigned>(d.Hkv)),
                                         dim3(static_cast<unsigned>((d.N + kRange1 - 1) / kRange1), nt, 1), rows,
                                         tfs, tk, a, st);
    }
    a.head_split = 0;
    const dim3 g(static_cast<unsigned>(a.n_ranges), nt, 1);
    return run_tok_passes_s<G, false>(g, g, rows, tfs, tk, a, st);
}

}  // namespace

int tok_range(const Derived& d)
{
    const int r = 128 * d.g;
    return r < 1024 ? r : 1024;
}

cudaError_t launch_select_tokens(const Derived& d, int mode, int64_t tok_begin, int64_t tok_end,
                                 const void* k, const KvPaging& pg, const float* fingerprints,
                                 const int32_t* unit_start,
                                 const int32_t* n_units, int32_t* sel, int32_t* sel_count,
                                 float* sel_scores, uint8_t* ws, uint64_t timeout_ns, cudaStream_t st)
{
    const WsLayout lay = ws_layout(d);
    TokArgs a;
    a.ut = Units{unit_start, n_units, mode == SCALE_MODE_PER_SUBCHUNK, d.N, d.L, static_cast<int>(d.M)};
    a.sc_begin = static_cast<int>(tok_begin / d.L);
    a.sc_end = static_cast<int>((tok_end + d.L - 1) / d.L);
    a.Hq = d.Hq;
    a.Hkv = d.Hkv;
    a.g = d.g;
    a.U = 128 / d.g;
    a.range = tok_range(d);
    a.n_ranges = static_cast<int>((d.N + a.range - 1) / a.range);
    a.N = static_cast<int>(d.N);
    a.n_sink = d.n_sink;
    a.n_local = d.n_local;
    a.head_split = 0;
    a.scale2 = d.sigma * 1.4426950408889634f;
    a.part = reinterpret_cast<float2*>(ws + lay.tok_part);
    a.stats = reinterpret_cast<const float2*>(ws + lay.stats);
    a.scores = sel_scores ? sel_scores : reinterpret_cast<float*>(ws + lay.scores);
    a.status = reinterpret_cast<int32_t*>(ws + kStatusOffset);
    a.timeout_ns = timeout_ns;
    a.pg = pg;
    const int max_units = a.sc_end - a.sc_begin;
    if (max_units <= 0) return cudaSuccess;

    auto* parts = reinterpret_cast<__nv_bfloat16*>(ws + lay.tok_split);
    CUtensorMap tf, tk;
    const uint64_t fdims[4] = {kHeadDim, static_cast<uint64_t>(d.M) * d.g, static_cast<uint64_t>(d.Hkv), 3};
    const uint32_t fbox[4] = {64, 128, 1, 1};
    if (!scale_host::make_dense_bf16_map(&tf, parts, 4, fdims, fbox) ||
        !scale_host::make_token_major_map(&tk, k, kHeadDim, d.Hkv, pg.page_table ? pg.pool_rows : d.N, 64, 64))
        return cudaErrorInvalidValue;

    k_tok_split<<<static_cast<unsigned>(max_units) * d.Hq, 128, 0, st>>>(a, fingerprints, parts, static_cast<int>(d.M));
    const int64_t rows = static_cast<int64_t>(max_units) * d.Hq;
    cudaError_t e = cudaSuccess;
    if (max_units <= kSmallUnits) {
        // few units (every call of the Algorithm 2 loop): 16 (unit, head) columns per tile
        CUtensorMap tfs;
        const uint32_t fbox_s[4] = {64, kNc, 1, 1};
        if (!scale_host::make_dense_bf16_map(&tfs, parts, 4, fdims, fbox_s)) return cudaErrorInvalidValue;
        const int tiles = (max_units + kNc / d.g - 1) / (kNc / d.g);
        switch (d.g) {
        case 1: e = run_tok_passes_s<1>(d, tiles, rows, tfs, tk, a, st); break;
        case 2: e = run_tok_passes_s<2>(d, tiles, rows, tfs, tk, a, st); break;
        case 3: e = run_tok_passes_s<3>(d, tiles, rows, tfs, tk, a, st); break;
        case 4: e = run_tok_passes_s<4>(d, tiles, rows, tfs, tk, a, st); break;
        case 5: e = run_tok_passes_s<5>(d, tiles, rows, tfs, tk, a, st); break;
        case 6: e = run_tok_passes_s<6>(d, tiles, rows, tfs, tk, a, st); break;
        case 7: e = run_tok_passes_s<7>(d, tiles, rows, tfs, tk, a, st); break;
        case 8: e = run_tok_passes_s<8>(d, tiles, rows, tfs, tk, a, st); break;
        default: return cudaErrorInvalidValue;
        }
        if (e == cudaSuccess) e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        const TopkScratch scratch{reinterpret_cast<int32_t*>(ws + lay.topk_hist),
                                  reinterpret_cast<int32_t*>(ws + lay.topk_state),
                                  reinterpret_cast<int2*>(ws + lay.topk_counts), topk_max_chunks(d)};
        return launch_topk(d, a.ut, a.sc_begin, a.sc_end, a.scores, sel, sel_count, st, nullptr, &scratch);
    }
    const int tiles_u = (max_units + a.U - 1) / a.U;
    const dim3 grid(static_cast<unsigned>(a.n_ranges), static_cast<unsigned>(tiles_u));
    switch (d.g) {
    case 1: e = run_tok_passes<1>(grid, rows, tf, tk, a, st); break;
    case 2: e = run_tok_passes<2>(grid, rows, tf, tk, a, st); break;
    case 3: e = run_tok_passes<3>(grid, rows, tf, tk, a, st); break;
    case 4: e = run_tok_passes<4>(grid, rows, tf, tk, a, st); break;
    case 5: e = run_tok_passes<5>(grid, rows, tf, tk, a, st); break;
    case 6: e = run_tok_passes<6>(grid, rows, tf, tk, a, st); break;
    case 7: e = run_tok_passes<7>(grid, rows, tf, tk, a, st); break;
    case 8: e = run_tok_passes<8>(grid, rows, tf, tk, a, st); break;
    default: return cudaErrorInvalidValue;
    }
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const TopkScratch scratch{reinterpret_cast<int32_t*>(ws + lay.topk_hist),
                              reinterpret_cast<int32_t*>(ws + lay.topk_state),
                              reinterpret_cast<int2*>(ws + lay.topk_counts), topk_max_chunks(d)};
    return launch_topk(d, a.ut, a.sc_begin, a.sc_end, a.scores, sel, sel_count, st, nullptr, &scratch);
}

}  // namespace scale
