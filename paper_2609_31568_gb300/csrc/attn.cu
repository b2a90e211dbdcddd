// attn.cu -- step (d) of the SCR prefill path: block-sparse causal attention
// over the cluster (Eq. 10, Sec. V-A3 "Sparse attention over the cluster").
//
// For a query row p of unit u = [s_u, e_u) the key set is
//   K(p) = D_u  U  [W_u, p],   D_u = ([0, n_sink) U selected blocks) n [0, W_u),
// W_u = max(0, s_u - n_local): the distant part D_u is shared by every row of
// the unit (the anchor-shared retrieval), the local part is the cluster-
// spanning window with the causal mask. Because D_u lies below W_u and the
// window starts at W_u, the two never overlap, and D_u is built from the sink
// range and each selected block clipped to [n_sink, W_u), so every key is
// visited once (the de-duplication of Sec. V-A3).
//
// Design (one CTA per work item = 128 query rows x 2 query heads of one KV head;
// with an odd number of query heads per KV head the last one of each group
// runs alone, as a CTA with one query tile):
//  - D_u is cut into 64-row segments; two segments form a 128-key tile. Each
//    segment is one TMA box per 64-column half of head_dim, so gathered blocks
//    land in shared memory in the 128-byte-swizzled K-major layout the tensor
//    cores read, with no copy through registers.
//  - warp 8 (one thread) issues TMA loads: both Q tiles once, then K and V
//    tiles into a 2-stage ring, K(t) and V(t - 1) on one barrier;
//  - warp 9 (one thread) issues tcgen05.mma: S_q = Q_q K^T into TMEM, and
//    O_q += P_q V with P read from TMEM (bf16, written over S_q). This thread
//    bounds the kernel: every barrier operation it runs between two MMA
//    groups leaves the tensor pipe idle, so it runs as few as it can (one
//    K/V wait, and per query tile one P wait, one fence and one commit per
//    key tile; the producer reuses the S-ready commits to free its stages);
//  - warps 0-3 and 4-7 run the online softmax of Q tile 0 and 1, one thread
//    per row (= TMEM lane), and the epilogue. The running max is raised only
//    when it grows by more than 8 (log2 units), so O is rescaled rarely; the
//    final normalisation uses the same max, which keeps the result exact.
//    Most tiles skip the row max altogether (see the fast path below).
//  - Every wait is bounded in wall time; on expiry the kernel records
//    SCALE_ERR_TIMEOUT, drains its in-flight copies and MMAs, frees TMEM and
//    returns.
#include <cuda_bf16.h>

#include "ptx_sm103.cuh"
#include "scale_internal.h"
#include "tma_host.h"

namespace scale {
namespace {

using namespace scale_ptx;

constexpr int kThreads = 320;
constexpr int kRows = 128;                    // query rows per Q tile
constexpr uint32_t kTileBytes = 128 * 128 * 2;  // one 128 x 128 bf16 tile
constexpr uint32_t kHalf = kTileBytes / 2;    // one 64-column half (128 rows x 128 B)
constexpr uint32_t kSegBytes = 64 * 128;      // one 64-row x 64-column box
constexpr float kRescaleThreshold = 8.0f;     // log2 units
constexpr float kFastSumLimit = 65536.0f;     // 2^16: largest tile sum kept on the fast path
// Softmax exponentials of column pair i go to the FMA pipe (exp2_poly2) when
// bit (i % 8) is set, else to the special-function unit. On sm_103 the
// special-function unit is not what bounds the softmax (moving any share of
// the exponentials only added issue slots in measurements), so none are moved
// by default.
#ifndef SCALE_SOFT_EXP_MASK
#define SCALE_SOFT_EXP_MASK 0x00
#endif
constexpr uint32_t kSoftExpMask = SCALE_SOFT_EXP_MASK;

// Dynamic shared memory map (offsets from the 1024-aligned base).
constexpr uint32_t kOffQ = 0;                          // 2 Q tiles
constexpr uint32_t kOffK = kOffQ + 2 * kTileBytes;     // 2 K stages
constexpr uint32_t kOffV = kOffK + 2 * kTileBytes;     // 2 V stages
constexpr uint32_t kOffSeg = kOffV + 2 * kTileBytes;   // int2 segment table
constexpr uint32_t kSmemBytes = kOffSeg + kMaxSegments * 8 + 1024;

struct AttnArgs {
    Units ut;
    int sc_begin, sc_end;
    int n_sc;       // sub-chunks in the token range
    int qb_per_sc;     // 128-row query blocks per sub-chunk
    int sc_per_chunk;  // sub-chunks per outer chunk
    int Hq, Hkv, g, pairs;
    int64_t N, nb;
    int B, k, n_sink, n_local;
    float scale_log2;
    const int32_t* sel;
    const int32_t* sel_count;
    const int32_t* tok_count;  // block size 1: [M] distant keys of each unit (packed)
    int slots;                 // block size 1: packed rows per (unit, KV head), a multiple of 128
    __nv_bfloat16* out;
    int32_t* status;
    uint64_t timeout_ns;
    KvPaging pg;
};

struct Barriers {
    uint64_t q_full;
    uint64_t kv_full[2];    // [t & 1]: K(t) and V(t - 1) landed (step T: V(T - 1) alone)
    uint64_t s_full[2][2];  // [q][t & 1]: S(t) of Q tile q ready (and every earlier MMA of the CTA done)
    uint64_t p_full[2];  // P of Q tile q written (128 arrivals)
    uint64_t o_full;     // last P.V of both tiles done
    uint64_t drain;
};

__device__ __forceinline__ void fail(volatile int* abort_flag, int32_t* status)
{
    *abort_flag = 1;
    record_status(status, SCALE_ERR_TIMEOUT);
}

// One iteration t (t & 1 = ST) of the MMA issue loop of a CTA with NQ (1 or 2)
// query tiles: wait for K(t) and V(t - 1), then per query tile wait for
// P(t - 1), issue O += P(t - 1) V(t - 1) and S = Q K(t)^T, and commit S-ready.
template <int NQ, int ST>
__device__ __forceinline__ bool mma_iteration(Barriers* bars, uint32_t tmem, uint64_t qdesc0, uint64_t kdesc0,
                                              uint64_t vdesc0, uint32_t id_qk, uint32_t id_pv, int t,
                                              uint64_t timeout_ns, const volatile int* abort_flag)
{
    // Descriptors of the two stages differ by kTileBytes >> 4 in the address field.
    constexpr uint64_t kStageStep = kTileBytes >> 4;
    const uint32_t ph = (t >> 1) & 1;
    if (!mbar_test(&bars->kv_full[ST], ph) && !mbar_wait_bounded(&bars->kv_full[ST], ph, timeout_ns, abort_flag))
        return false;
    // TMA data is ordered by the barrier's transaction count; from t = 1
    // the fence after the P wait below precedes every MMA of the iteration.
    if (t == 0) tc_fence_after();
#pragma unroll
    for (int qt = 0; qt < NQ; ++qt) {
        if (t > 0) {
            if (!mbar_wait_bounded(&bars->p_full[qt], ST ^ 1, timeout_ns, abort_flag)) return false;
            tc_fence_after();
            mma_ts_k128<2048>(tmem + qt * 256 + 128, tmem + qt * 256, vdesc0 + (ST ^ 1) * kStageStep, id_pv,
                              t > 1 ? 1u : 0u);
        }
        mma_ss_k128<kHalf>(tmem + qt * 256, qdesc0 + qt * kStageStep, kdesc0 + ST * kStageStep, id_qk, 0u);
        mma_commit(&bars->s_full[qt][ST]);
    }
    return true;
}

// The MMA issue loop, run by one thread: T iterations (two per trip, so the
// stage indices are constants), then the last P.V and the O-ready commit.
// This thread is the critical path: NQ is a compile-time constant and all
// state is held in registers. Returns false when a wait ran out or the
// kernel was aborted.
template <int NQ>
__device__ __forceinline__ bool mma_issue_loop(Barriers* bars, uint32_t tmem, uint64_t qdesc0, uint64_t kdesc0,
                                               uint64_t vdesc0, uint32_t id_qk, uint32_t id_pv, int T,
                                               uint64_t timeout_ns, const volatile int* abort_flag)
{
    constexpr uint64_t kStageStep = kTileBytes >> 4;
    int t = 0;
    for (; t + 1 < T; t += 2) {
        if (!mma_iteration<NQ, 0>(bars, tmem, qdesc0, kdesc0, vdesc0, id_qk, id_pv, t, timeout_ns, abort_flag) ||
            !mma_iteration<NQ, 1>(bars, tmem, qdesc0, kdesc0, vdesc0, id_qk, id_pv, t + 1, timeout_ns, abort_flag))
            return false;
    }
    if (t < T && !mma_iteration<NQ, 0>(bars, tmem, qdesc0, kdesc0, vdesc0, id_qk, id_pv, t, timeout_ns, abort_flag))
        return false;
    if (!mbar_wait_bounded(&bars->kv_full[T & 1], (T >> 1) & 1, timeout_ns, abort_flag)) return false;
#pragma unroll
    for (int qt = 0; qt < NQ; ++qt) {
        if (!mbar_wait_bounded(&bars->p_full[qt], (T - 1) & 1, timeout_ns, abort_flag)) return false;
        tc_fence_after();
        mma_ts_k128<2048>(tmem + qt * 256 + 128, tmem + qt * 256, vdesc0 + ((T - 1) & 1) * kStageStep, id_pv,
                          T > 1 ? 1u : 0u);
    }
    mma_commit(&bars->o_full);
    return true;
}

// TOK: block size 1. The distant keys and values of each (unit, KV head)
// were packed by k_tok_pack into contiguous rows [M * H_kv][slots][128]
// (zero rows after the last one), so their tiles are plain TMA boxes of the
// maps tpk / tpv, like the window's.
template <bool TOK>
__global__ void __launch_bounds__(kThreads, 1)
k_sparse_attn(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tk,
              const __grid_constant__ CUtensorMap tv, const __grid_constant__ CUtensorMap tpk,
              const __grid_constant__ CUtensorMap tpv, const AttnArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ Barriers bars;
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    __shared__ int s_nseg;

    // ---- work item: a 128-row query block of one sub-chunk and a pair of
    // query heads. The grid holds exactly the blocks of the sub-chunks in
    // range (no idle CTAs whatever the clustering), outer chunk by outer
    // chunk, and within a chunk KV head by KV head, so the CTAs resident at
    // a time share the K/V rows of one or two KV heads of one cluster (a few
    // MB, which L2 keeps); for each KV head the chunk's last query block
    // comes first, which issues the heaviest rows (longest window) first. ----
    const int per_chunk = a.sc_per_chunk * a.qb_per_sc;  // query blocks of a full chunk
    const int per_chunk_ctas = per_chunk * a.Hkv * a.pairs;
    const int c = static_cast<int>(blockIdx.x) / per_chunk_ctas;
    const int sc0 = a.sc_begin + c * a.sc_per_chunk;
    const int n_sc = (a.sc_end - sc0 < a.sc_per_chunk) ? a.sc_end - sc0 : a.sc_per_chunk;
    const int n_qb = n_sc * a.qb_per_sc;  // query blocks of this chunk
    int rem = static_cast<int>(blockIdx.x) - c * per_chunk_ctas;
    const int kvh = rem / (n_qb * a.pairs);
    rem -= kvh * n_qb * a.pairs;
    const int qb = rem / a.pairs;
    const int h0 = kvh * a.g + 2 * (rem - qb * a.pairs);
    const int nq = (h0 + 1 < (kvh + 1) * a.g) ? 2 : 1;  // query tiles (heads) of this CTA
    const int idx = n_qb - 1 - qb;
    if (idx < 0 || kvh >= a.Hkv) return;
    const int sc = sc0 + idx / a.qb_per_sc;
    const int u = unit_of_subchunk(a.ut, sc);
    int anchor;
    int64_t s_u, e_u;
    unit_range(a.ut, u, &anchor, &s_u, &e_u);
    const int64_t sc_lo = static_cast<int64_t>(sc) * a.ut.L;
    const int64_t sc_hi = (sc_lo + a.ut.L < e_u) ? sc_lo + a.ut.L : e_u;
    const int64_t q0 = sc_lo + static_cast<int64_t>(kRows) * (idx % a.qb_per_sc);
    if (q0 >= sc_hi) return;
    const int64_t q_end = (q0 + kRows < sc_hi) ? q0 + kRows : sc_hi;
    const int64_t W = (s_u - a.n_local > 0) ? s_u - a.n_local : 0;
    const int n_lt = static_cast<int>((q_end - W + 127) / 128);

    uint8_t* smem = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
    int2* seg = reinterpret_cast<int2*>(smem + kOffSeg);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        abort_flag = 0;
        mbar_init(&bars.q_full, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars.kv_full[i], 1);
            mbar_init(&bars.s_full[i][0], 1);
            mbar_init(&bars.s_full[i][1], 1);
            mbar_init(&bars.p_full[i], 128);
        }
        mbar_init(&bars.o_full, 1);
        mbar_init(&bars.drain, 1);
        fence_barrier_init();
    }
    if (warp == 9) {
        tmem_alloc(&tmem_slot, 512);
        tmem_relinquish();
    }
    if (TOK && warp == 8) {
        if (lane == 0) {
            int n = a.tok_count[u];
            n = n < 0 ? 0 : (n > a.slots ? a.slots : n);
            s_nseg = n;  // distant tokens (not segments) in this mode
        }
    } else if (warp == 8) {
        // Distant segments: the sinks, then each selected block clipped to
        // [n_sink, W); 64 rows at most per segment.
        const int64_t sink_end = a.n_sink < W ? a.n_sink : W;
        const int n_sink_seg = static_cast<int>((sink_end + 63) / 64);
        for (int i = lane; i < n_sink_seg; i += 32) {
            const int64_t t0 = 64ll * i;
            seg[i] = make_int2(static_cast<int>(t0), static_cast<int>(sink_end - t0 < 64 ? sink_end - t0 : 64));
        }
        int base = n_sink_seg;
        int cnt = a.sel_count[u];
        cnt = cnt < 0 ? 0 : (cnt > a.k ? a.k : cnt);
        const int32_t* sl = a.sel + static_cast<int64_t>(u) * a.k;
        bool overflow = false;
        for (int c0 = 0; c0 < cnt; c0 += 32) {
            const int i = c0 + lane;
            int nseg = 0;
            int64_t lo = 0, hi = 0;
            if (i < cnt) {
                const int64_t b = sl[i];
                const int64_t prev = i > 0 ? sl[i - 1] : -1;
                if (b >= 0 && b < a.nb && b > prev) {
                    lo = b * a.B > a.n_sink ? b * a.B : a.n_sink;
                    hi = (b + 1) * a.B < W ? (b + 1) * a.B : W;
                    if (hi > lo) nseg = static_cast<int>((hi - lo + 63) / 64);
                }
            }
            int incl = nseg;
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                if (lane >= o) incl += y;
            }
            const int off = base + incl - nseg;
            if (off + nseg > kMaxSegments - 1) overflow = true;
            else
                for (int m = 0; m < nseg; ++m) {
                    const int64_t t0 = lo + 64ll * m;
                    seg[off + m] = make_int2(static_cast<int>(t0), static_cast<int>(hi - t0 < 64 ? hi - t0 : 64));
                }
            base += __shfl_sync(0xFFFFFFFFu, incl, 31);
        }
        overflow = __any_sync(0xFFFFFFFFu, overflow);
        if (lane == 0) {
            if (overflow) {
                record_status(a.status, SCALE_ERR_DEVICE);
                base = 0;
            }
            if (base & 1) seg[base] = make_int2(0, 0);
            s_nseg = base;
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    const int n_dt = TOK ? (s_nseg + 127) / 128 : (s_nseg + 1) / 2;
    const int T = n_dt + n_lt;

    if (warp == 8) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&tq);
            tma_prefetch_desc(&tk);
            tma_prefetch_desc(&tv);
            if (TOK) {
                tma_prefetch_desc(&tpk);
                tma_prefetch_desc(&tpv);
            }
            mbar_arrive_expect_tx(&bars.q_full, nq * kTileBytes);
            for (int qt = 0; qt < nq; ++qt)
                for (int hf = 0; hf < 2; ++hf)
                    tma_load_3d(smem + kOffQ + qt * kTileBytes + hf * kHalf, &tq, &bars.q_full,
                                hf * 64, h0 + qt, static_cast<int32_t>(q0));
            const int32_t prow = u * a.Hkv + kvh;  // packed (unit, KV head) plane
            // Step t (0..T) loads K(t) and V(t - 1) on kv_full[t & 1]; both stages
            // they reuse were last read by MMAs of iteration t - 2 (Q K^T of K(t - 2),
            // P.V of V(t - 3)), which the S-ready commit of the CTA's last query
            // tile in that iteration covers.
            uint64_t* const s_last = bars.s_full[nq - 1];
            int issued0 = 0, issued1 = 0;
            int32_t pa = 0, pb = 0;  // TMA rows of tile t - 1 (its V goes out at step t)
            bool p_packed = false;
            int32_t p_ta = 0;
            for (int t = 0; t <= T && !abort_flag; ++t) {
                const int st = t & 1;
                if (t >= 2 && !mbar_wait_bounded(&s_last[st], ((t - 2) >> 1) & 1, a.timeout_ns, &abort_flag)) {
                    fail(&abort_flag, a.status);
                    break;
                }
                const bool has_k = t < T, has_v = t >= 1;
                mbar_arrive_expect_tx(&bars.kv_full[st], (has_k ? kTileBytes : 0u) + (has_v ? kTileBytes : 0u));
                if (st) ++issued1; else ++issued0;
                if (has_v) {
                    uint8_t* vd = smem + kOffV + ((t - 1) & 1) * kTileBytes;
                    for (int hf = 0; hf < 2; ++hf) {
                        if (p_packed) {
                            tma_load_3d(vd + hf * kHalf, &tpv, &bars.kv_full[st], hf * 64, p_ta, prow);
                        } else {
                            tma_load_3d(vd + hf * kHalf, &tv, &bars.kv_full[st], hf * 64, kvh, pa);
                            tma_load_3d(vd + hf * kHalf + kSegBytes, &tv, &bars.kv_full[st], hf * 64, kvh, pb);
                        }
                    }
                }
                if (has_k) {
                    const bool packed = TOK && t < n_dt;
                    int32_t ta, tb;
                    if (packed) {
                        ta = 128 * t;
                        tb = 0;
                    } else if (t < n_dt) {
                        ta = seg[2 * t].x;
                        tb = seg[2 * t + 1].x;
                    } else {
                        ta = static_cast<int32_t>(W + 128ll * (t - n_dt));
                        tb = ta + 64;
                    }
                    // 64-row boxes: every one lies inside one KV page
                    const int32_t ra = packed ? 0 : kv_row_tma(a.pg, ta);
                    const int32_t rb = packed ? 0 : kv_row_tma(a.pg, tb);
                    uint8_t* kd = smem + kOffK + st * kTileBytes;
                    for (int hf = 0; hf < 2; ++hf) {
                        if (packed) {
                            tma_load_3d(kd + hf * kHalf, &tpk, &bars.kv_full[st], hf * 64, ta, prow);
                        } else {
                            tma_load_3d(kd + hf * kHalf, &tk, &bars.kv_full[st], hf * 64, kvh, ra);
                            tma_load_3d(kd + hf * kHalf + kSegBytes, &tk, &bars.kv_full[st], hf * 64, kvh, rb);
                        }
                    }
                    pa = ra;
                    pb = rb;
                    p_packed = packed;
                    p_ta = ta;
                }
            }
            if (abort_flag) {
                // Drain: wait (bounded, ignoring the abort flag) for the last
                // phase of every buffer that received copies.
                mbar_wait_bounded(&bars.q_full, 0, a.timeout_ns, nullptr);
                if (issued0) mbar_wait_bounded(&bars.kv_full[0], (issued0 - 1) & 1, a.timeout_ns, nullptr);
                if (issued1) mbar_wait_bounded(&bars.kv_full[1], (issued1 - 1) & 1, a.timeout_ns, nullptr);
            }
        }
    } else if (warp == 9) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t id_qk = idesc_bf16_f32(128, 128, 0);
            const uint32_t id_pv = idesc_bf16_f32(128, 128, 1);
            const uint32_t q_base = smem_addr(smem + kOffQ);
            const uint32_t k_base = smem_addr(smem + kOffK);
            const uint32_t v_base = smem_addr(smem + kOffV);
            bool ok = mbar_wait_bounded(&bars.q_full, 0, a.timeout_ns, &abort_flag);
            const uint64_t qdesc0 = sdesc_sw128(q_base, 16, 1024);
            const uint64_t kdesc0 = sdesc_sw128(k_base, 16, 1024);
            const uint64_t vdesc0 = sdesc_sw128(v_base, kHalf, 1024);
            if (ok)
                ok = nq == 2 ? mma_issue_loop<2>(&bars, tmem, qdesc0, kdesc0, vdesc0, id_qk, id_pv, T, a.timeout_ns,
                                                 &abort_flag)
                             : mma_issue_loop<1>(&bars, tmem, qdesc0, kdesc0, vdesc0, id_qk, id_pv, T, a.timeout_ns,
                                                 &abort_flag);
            if (!ok) {
                fail(&abort_flag, a.status);
                // Drain: every MMA issued so far completes before TMEM is freed.
                mma_commit(&bars.drain);
                mbar_wait_bounded(&bars.drain, 0, a.timeout_ns, nullptr);
            }
        }
    } else if ((warp >> 2) < nq) {
        // ------------------------------------------------------------ softmax + epilogue
        const int qt = warp >> 2;
        const int quarter = warp & 3;
        const int r = quarter * 32 + lane;
        const int64_t p = q0 + r;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
        const uint32_t s_addr = lane_base + qt * 256;
        const uint32_t o_addr = s_addr + 128;
        float m_run = -INFINITY, l_run = 0.f;
        bool ok = true;
        // S row of tile t: four 32-column TMEM loads in flight, one wait, then
        // the keys outside the row's key set set to -inf: column c < 64 when
        // c >= lim_a, column c >= 64 when c - 64 >= lim_b.
        auto load_s = [&](uint32_t (&sr)[128], int lim_a, int lim_b) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                tmem_ld32(s_addr + c * 32, *reinterpret_cast<uint32_t(*)[32]>(&sr[c * 32]));
            tmem_ld_wait();
            float* s = reinterpret_cast<float*>(sr);
            if (lim_a < 64 || lim_b < 64) {
#pragma unroll
                for (int c = 0; c < 128; ++c)
                    if (c < 64 ? c >= lim_a : c - 64 >= lim_b) s[c] = -INFINITY;
            }
        };
        // p = 2^(s * scale_log2 - m) for keys [64 h, 64 h + 64): packed FMA, then
        // the exponential, packed to bf16 pairs in pk; returns the sum of the p.
        auto exp_half = [&](const float* s, int h, float neg_m, uint32_t (&pk)[32]) {
            float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                float x0, x1;
                ffma2(x0, x1, s[h * 64 + 2 * i], s[h * 64 + 2 * i + 1], a.scale_log2, a.scale_log2, neg_m,
                      neg_m);
                if ((kSoftExpMask >> (i & 7)) & 1u) {
                    exp2_poly2(x0, x1, x0, x1);
                } else {
                    x0 = ex2(x0);
                    x1 = ex2(x1);
                }
                const int j = (i & 3) * 2;
                fadd2(acc[j], acc[j + 1], acc[j], acc[j + 1], x0, x1);
                pk[i] = pack_bf16x2(x0, x1);
            }
            return ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
        };
        for (int t = 0; t < T; ++t) {
            // tcgen05.ld/st are warp-collective: the outcome must be warp-uniform.
            const bool got = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(&bars.s_full[qt][t & 1], (t >> 1) & 1, a.timeout_ns, &abort_flag));
            if (!got) { ok = false; break; }
            tc_fence_after();
            // Mask limits of tile t (128: nothing masked).
            int lim_a = 128, lim_b = 128;
            if (TOK && t < n_dt) {
                const int lim = s_nseg - 128 * t;  // packed rows past the list are zero padding
                if (lim < 128) {
                    lim_a = lim < 0 ? 0 : lim;
                    lim_b = lim_a - 64;
                }
            } else if (t < n_dt) {
                lim_a = seg[2 * t].y;
                lim_b = seg[2 * t + 1].y;
            } else {
                const int64_t kb = W + 128ll * (t - n_dt);
                if (kb + 127 > q0) {
                    const int64_t lim = p - kb + 1;  // keys kb + c with c >= lim are in the future
                    lim_a = lim < 0 ? 0 : (lim > 128 ? 128 : static_cast<int>(lim));
                    lim_b = lim_a - 64;
                }
            }
            // Fast path: the exponentials are taken against the running max as it
            // stands, without the row max. The max only matters when the tile
            // outgrows m_run by more than the raise threshold, and the sum shows
            // it: a sum above 2^16 over 128 keys needs a term above 2^9, i.e. a
            // logit more than 9 (log2 units) above m_run. Below that every p is
            // at most 2^16, far inside the fp32 and bf16 ranges, so m_run may
            // stay; a sum that is inf or NaN fails the test as well. The first
            // tile (m_run = -inf) and every failed tile take the exact path (row
            // max, raise, O rescale) on a fresh copy of S: nothing has been
            // stored over it yet.
            bool exact = !__all_sync(0xFFFFFFFFu, m_run != -INFINITY);
            float sum;
#pragma unroll 1
            for (;;) {
                uint32_t sr[128];
                load_s(sr, lim_a, lim_b);
                const float* s = reinterpret_cast<const float*>(sr);
                if (exact) {
                    // Row max: eight independent three-input max chains.
                    float mx8[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) mx8[i] = s[i];
#pragma unroll
                    for (int c = 8; c < 120; c += 16)
#pragma unroll
                        for (int i = 0; i < 8; ++i) mx8[i] = fmax3(mx8[i], s[c + 2 * i], s[c + 2 * i + 1]);
#pragma unroll
                    for (int i = 0; i < 8; ++i) mx8[i] = fmaxf(mx8[i], s[120 + i]);
                    const float mx = fmax3(fmax3(mx8[0], mx8[1], mx8[2]), fmax3(mx8[3], mx8[4], mx8[5]),
                                           fmaxf(mx8[6], mx8[7]));
                    const float m_new = fmaxf(m_run, mx * a.scale_log2);
                    const bool raise = m_new > m_run + kRescaleThreshold;
                    // The O rescale goes through warp-collective TMEM loads and stores,
                    // so the branch is taken by the whole warp when any row needs it;
                    // rows that do not keep their max and scale by 1.
                    if (__any_sync(0xFFFFFFFFu, raise)) {
                        const float alpha = raise ? ex2(m_run - m_new) : 1.0f;
                        l_run *= alpha;
                        if (t > 0) {
#pragma unroll 1
                            for (int c = 0; c < 8; ++c) {
                                uint32_t v[16];
                                tmem_ld16(o_addr + c * 16, v);
                                tmem_ld_wait();
#pragma unroll
                                for (int i = 0; i < 16; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * alpha);
                                tmem_st16(o_addr + c * 16, v);
                            }
                        }
                        if (raise) m_run = m_new;
                    }
                }
                const float neg_m = (m_run == -INFINITY) ? 0.f : -m_run;
                uint32_t pk[2][32];
                sum = exp_half(s, 0, neg_m, pk[0]);
                sum += exp_half(s, 1, neg_m, pk[1]);
                if (!exact && __any_sync(0xFFFFFFFFu, !(sum <= kFastSumLimit))) {
                    exact = true;
                    continue;
                }
                tmem_st32(s_addr, pk[0]);
                tmem_st32(s_addr + 32, pk[1]);
                break;
            }
            l_run += sum;
            tmem_st_wait();
            tc_fence_before();
            mbar_arrive(&bars.p_full[qt]);
        }
        bool go = __all_sync(0xFFFFFFFFu, ok && !abort_flag);
        if (go) go = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(&bars.o_full, 0, a.timeout_ns, &abort_flag));
        if (go) {
            tc_fence_after();
            const float inv_l = l_run > 0.f ? 1.0f / l_run : 0.f;
            const bool store = p < q_end;
            uint4* dst = reinterpret_cast<uint4*>(a.out + (p * a.Hq + h0 + qt) * static_cast<int64_t>(kHeadDim));
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t v[32];
                tmem_ld32(o_addr + c * 32, v);
                tmem_ld_wait();
                if (store) {
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        dst[c * 4 + i] = make_uint4(
                            pack_bf16x2(__uint_as_float(v[8 * i + 0]) * inv_l, __uint_as_float(v[8 * i + 1]) * inv_l),
                            pack_bf16x2(__uint_as_float(v[8 * i + 2]) * inv_l, __uint_as_float(v[8 * i + 3]) * inv_l),
                            pack_bf16x2(__uint_as_float(v[8 * i + 4]) * inv_l, __uint_as_float(v[8 * i + 5]) * inv_l),
                            pack_bf16x2(__uint_as_float(v[8 * i + 6]) * inv_l, __uint_as_float(v[8 * i + 7]) * inv_l));
                }
            }
        } else {
            fail(&abort_flag, a.status);
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// Block size 1, step 1 of 2: the distant list of every unit, one CTA per
// unit: the sinks [0, min(n_sink, W_u)), then every selected token in
// [n_sink, W_u) larger than the entry before it (each key once, ascending).
// The selected entries are compacted in order by one block-wide scan: each
// thread takes kListPer consecutive entries.
constexpr int kListThreads = 1024;
constexpr int kListPer = 8;
__global__ void __launch_bounds__(kListThreads) k_tok_lists(Units ut, int sc_begin, int sc_end, int n_sink,
                                                            int n_local, int k, const int32_t* __restrict__ sel,
                                                            const int32_t* __restrict__ sel_count,
                                                            int32_t* __restrict__ list, int32_t* __restrict__ count,
                                                            int slots)
{
    __shared__ int s_warp[kListThreads / 32];
    const int u = unit_lower_bound(ut, sc_begin) + static_cast<int>(blockIdx.x);
    if (u >= unit_lower_bound(ut, sc_end)) return;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int anchor;
    int64_t s_u, e_u;
    unit_range(ut, u, &anchor, &s_u, &e_u);
    const int64_t W = (s_u - n_local > 0) ? s_u - n_local : 0;
    int32_t* out = list + static_cast<int64_t>(u) * slots;
    const int n_s = static_cast<int>(n_sink < W ? n_sink : W);
    for (int i = tid; i < n_s; i += kListThreads) out[i] = i;
    int cnt = sel_count[u];
    cnt = cnt < 0 ? 0 : (cnt > k ? k : cnt);
    const int32_t* sl = sel + static_cast<int64_t>(u) * k;
    int base = n_s;
    for (int c0 = 0; c0 < cnt; c0 += kListThreads * kListPer) {
        const int i0 = c0 + tid * kListPer;
        int32_t tok[kListPer];
        int prev = (i0 > 0 && i0 - 1 < cnt) ? sl[i0 - 1] : -1;
        unsigned valid = 0u;
#pragma unroll
        for (int j = 0; j < kListPer; ++j) {
            const int i = i0 + j;
            tok[j] = i < cnt ? sl[i] : -1;
            if (i < cnt && tok[j] >= n_sink && tok[j] < W && tok[j] > prev) valid |= 1u << j;
            if (i < cnt) prev = tok[j];
        }
        const int mine = __popc(valid);
        int incl = mine;
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) s_warp[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            const int x = s_warp[lane];
            int xi = x;
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xFFFFFFFFu, xi, o);
                if (lane >= o) xi += y;
            }
            s_warp[lane] = xi - x;  // exclusive prefix of the warps
        }
        __syncthreads();
        int pos = base + s_warp[warp] + incl - mine;
#pragma unroll
        for (int j = 0; j < kListPer; ++j)
            if ((valid >> j) & 1u) out[pos++] = tok[j];
        const int total = __shfl_sync(0xFFFFFFFFu, incl, 31);
        __syncthreads();
        // the block total: the last warp's exclusive prefix plus its total
        if (tid == kListThreads - 1) s_warp[0] = s_warp[warp] + total;
        __syncthreads();
        base += s_warp[0];
        __syncthreads();
    }
    if (tid == 0) count[u] = base;
}

// Block size 1, step 2 of 2: copy the listed K and V rows of unit u
// (blockIdx.x) and KV head blockIdx.y, slots [256 z, 256 z + 256) with
// z = blockIdx.z, into contiguous rows [M * H_kv][slots][128]; slots past the
// list up to the next multiple of 128 are written as zeros.
constexpr int kPackSlots = 256;
__global__ void __launch_bounds__(256) k_tok_pack(Units ut, int sc_begin, int sc_end, int Hkv, KvPaging pg,
                                                  const int32_t* __restrict__ list,
                                                  const int32_t* __restrict__ count,
                                                  const uint4* __restrict__ kin, const uint4* __restrict__ vin,
                                                  uint4* __restrict__ kout, uint4* __restrict__ vout, int slots)
{
    const int u = unit_lower_bound(ut, sc_begin) + static_cast<int>(blockIdx.x);
    if (u >= unit_lower_bound(ut, sc_end)) return;
    const int kvh = blockIdx.y;
    int n = count[u];
    n = n < 0 ? 0 : (n > slots ? slots : n);
    const int n_pad = (n + 127) / 128 * 128;
    const int s0 = static_cast<int>(blockIdx.z) * kPackSlots;
    const int s1 = (s0 + kPackSlots < n_pad) ? s0 + kPackSlots : n_pad;
    if (s0 >= s1) return;
    const int32_t* lu = list + static_cast<int64_t>(u) * slots;
    const int64_t plane = (static_cast<int64_t>(u) * Hkv + kvh) * slots * 16;  // 16-byte chunks
    const uint4 zero = make_uint4(0, 0, 0, 0);
    for (int i = s0 * 16 + static_cast<int>(threadIdx.x); i < s1 * 16; i += blockDim.x) {
        const int slot = i >> 4, c = i & 15;
        uint4 kx = zero, vx = zero;
        const int64_t row = slot < n ? kv_row(pg, lu[slot]) : -1;  // -1: zeros
        if (row >= 0) {
            const int64_t src = (row * Hkv + kvh) * 16 + c;
            kx = kin[src];
            vx = vin[src];
        }
        kout[plane + i] = kx;
        vout[plane + i] = vx;
    }
}

// Bounded-wait self-check: wait on a barrier nothing arrives at.
__global__ void k_wait_selftest(int32_t* status, uint64_t timeout_ns)
{
    __shared__ uint64_t bar;
    __shared__ volatile int never;
    if (threadIdx.x == 0) {
        never = 0;
        mbar_init(&bar, 1);
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0 && !mbar_wait_bounded(&bar, 0, timeout_ns, &never))
        record_status(status, SCALE_ERR_TIMEOUT);
}

}  // namespace

int tok_slots(const Derived& d)
{
    return (d.n_sink + d.k + 127) / 128 * 128;
}

int64_t max_distant_segments(const Derived& d)
{
    // ceil(n_sink / 64) sink segments, at most ceil(B / 64) per selected block,
    // plus one pad segment.
    return (d.n_sink + 63) / 64 + static_cast<int64_t>(d.k) * ((d.B + 63) / 64) + 1;
}

cudaError_t launch_sparse_prefill(const Derived& d, int mode, int64_t tok_begin, int64_t tok_end,
                                  const void* q, const void* k, const void* v, const KvPaging& pg,
                                  const int32_t* unit_start, const int32_t* n_units,
                                  const int32_t* sel_blocks, const int32_t* sel_count, void* out,
                                  uint8_t* ws, uint64_t timeout_ns, cudaStream_t st)
{
    CUtensorMap tq, tk, tv, tpk, tpv;
    if (!scale_host::make_token_major_map(&tq, q, kHeadDim, d.Hq, d.N, 64, 128) ||
        !scale_host::make_token_major_map(&tk, k, kHeadDim, d.Hkv, pg.page_table ? pg.pool_rows : d.N, 64, 64) ||
        !scale_host::make_token_major_map(&tv, v, kHeadDim, d.Hkv, pg.page_table ? pg.pool_rows : d.N, 64, 64))
        return cudaErrorInvalidValue;
    const bool tok = d.B == 1;
    const WsLayout lay = ws_layout(d);
    const int slots = tok_slots(d);
    if (tok) {
        // packed distant rows [M * H_kv][slots][128], boxes of 64 x 128 rows
        const uint64_t pdims[3] = {kHeadDim, static_cast<uint64_t>(slots), static_cast<uint64_t>(d.M) * d.Hkv};
        const uint32_t pbox[3] = {64, 128, 1};
        if (!scale_host::make_dense_bf16_map(&tpk, ws + lay.tok_pack_k, 3, pdims, pbox) ||
            !scale_host::make_dense_bf16_map(&tpv, ws + lay.tok_pack_v, 3, pdims, pbox))
            return cudaErrorInvalidValue;
    } else {
        tpk = tk;
        tpv = tv;
    }

    AttnArgs a;
    a.ut = Units{unit_start, n_units, mode == SCALE_MODE_PER_SUBCHUNK, d.N, d.L, static_cast<int>(d.M)};
    a.sc_begin = static_cast<int>(tok_begin / d.L);
    a.sc_end = static_cast<int>((tok_end + d.L - 1) / d.L);
    a.n_sc = a.sc_end - a.sc_begin;
    if (a.n_sc <= 0) return cudaSuccess;
    a.qb_per_sc = static_cast<int>((d.L + kRows - 1) / kRows);
    a.sc_per_chunk = d.per_outer;
    a.Hq = d.Hq;
    a.Hkv = d.Hkv;
    a.g = d.g;
    a.pairs = (d.g + 1) / 2;  // an odd group's last head runs alone
    a.N = d.N;
    a.nb = d.nb;
    a.B = d.B;
    a.k = d.k;
    a.n_sink = d.n_sink;
    a.n_local = d.n_local;
    a.scale_log2 = d.attn_scale * 1.4426950408889634f;
    a.sel = sel_blocks;
    a.sel_count = sel_count;
    a.tok_count = tok ? reinterpret_cast<const int32_t*>(ws + lay.tok_count) : nullptr;
    a.slots = slots;
    a.out = static_cast<__nv_bfloat16*>(out);
    a.status = reinterpret_cast<int32_t*>(ws + kStatusOffset);
    a.timeout_ns = timeout_ns;
    a.pg = pg;

    if (tok) {
        int32_t* list = reinterpret_cast<int32_t*>(ws + lay.tok_list);
        int32_t* cnt = const_cast<int32_t*>(a.tok_count);
        k_tok_lists<<<a.n_sc, kListThreads, 0, st>>>(a.ut, a.sc_begin, a.sc_end, d.n_sink, d.n_local, d.k, sel_blocks,
                                           sel_count, list, cnt, slots);
        k_tok_pack<<<dim3(a.n_sc, d.Hkv, (slots + kPackSlots - 1) / kPackSlots), 256, 0, st>>>(
            a.ut, a.sc_begin, a.sc_end, d.Hkv, pg, list, cnt, static_cast<const uint4*>(k),
            static_cast<const uint4*>(v), reinterpret_cast<uint4*>(ws + lay.tok_pack_k),
            reinterpret_cast<uint4*>(ws + lay.tok_pack_v), slots);
    }
    auto kern = tok ? k_sparse_attn<true> : k_sparse_attn<false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kSmemBytes));
    if (e != cudaSuccess) return e;
    const int64_t grid = static_cast<int64_t>(a.n_sc) * a.qb_per_sc * d.Hkv * a.pairs;
    if (grid <= 0 || grid > 0x7FFFFFFFll) return cudaErrorInvalidConfiguration;
    kern<<<static_cast<unsigned>(grid), kThreads, kSmemBytes, st>>>(tq, tk, tv, tpk, tpv, a);
    return cudaGetLastError();
}

cudaError_t launch_wait_selftest(uint8_t* ws, uint64_t timeout_ns, cudaStream_t st)
{
    k_wait_selftest<<<1, 32, 0, st>>>(reinterpret_cast<int32_t*>(ws + kStatusOffset), timeout_ns);
    return cudaGetLastError();
}

}  // namespace scale
