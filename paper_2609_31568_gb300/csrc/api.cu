// api.cu -- the extern "C" boundary of libscale: argument validation, the
// workspace layout, the launch of each step on the caller's stream, and the
// end-to-end call that works from host buffers.
#include <atomic>
#include <cmath>
#include <vector>

#include "scale_internal.h"

namespace scale {

static std::atomic<uint64_t> g_timeout_ns{4000000000ull};

int derive(const scale_params_t* p, Derived* d)
{
    if (!p || !d) return SCALE_ERR_INVALID_ARG;
    if (p->num_q_heads <= 0 || p->num_kv_heads <= 0 || p->num_q_heads % p->num_kv_heads)
        return SCALE_ERR_INVALID_ARG;
    if (p->head_dim != kHeadDim) return SCALE_ERR_UNSUPPORTED;
    if (p->n_tokens <= 0 || p->sub_chunk <= 0 || p->max_cluster_subchunks <= 0 ||
        p->outer_chunk < 0 || p->block_size <= 0 || p->top_k < 0 || p->n_sink < 0 ||
        p->n_local < 0)
        return SCALE_ERR_INVALID_ARG;
    if (std::isnan(p->theta) || !std::isfinite(p->select_scale) || !std::isfinite(p->attn_scale) ||
        p->attn_scale < 0.f)
        return SCALE_ERR_INVALID_ARG;
    const int64_t L_outer = p->outer_chunk ? p->outer_chunk
                                           : static_cast<int64_t>(p->max_cluster_subchunks) * p->sub_chunk;
    if (L_outer % p->sub_chunk) return SCALE_ERR_INVALID_ARG;
    const int g = p->num_q_heads / p->num_kv_heads;
    if (g > 32 || p->num_kv_heads > 64) return SCALE_ERR_UNSUPPORTED;
    if (p->n_tokens >= (1ll << 31) - 256) return SCALE_ERR_UNSUPPORTED;
    d->N = p->n_tokens;
    d->Hq = p->num_q_heads;
    d->Hkv = p->num_kv_heads;
    d->g = g;
    d->dh = p->head_dim;
    d->L = p->sub_chunk;
    d->S_max = p->max_cluster_subchunks;
    d->per_outer = static_cast<int>(L_outer / p->sub_chunk);
    d->B = p->block_size;
    d->k = p->top_k;
    d->n_sink = p->n_sink;
    d->n_local = p->n_local;
    d->M = (d->N + d->L - 1) / d->L;
    d->nb = (d->N + d->B - 1) / d->B;
    d->D = d->Hq * kHeadDim;
    d->fp_groups = (d->D / 8 + 31) / 32;  // 32 sixteen-byte columns per fingerprint CTA
    d->theta = p->theta;
    d->sigma = p->select_scale;
    d->attn_scale = p->attn_scale > 0.f ? p->attn_scale : 1.0f / std::sqrt(static_cast<float>(kHeadDim));
    return SCALE_OK;
}

WsLayout ws_layout(const Derived& d)
{
    WsLayout w{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t at = off;
        off = align_up(off + bytes, kAlign);
        return at;
    };
    w.status = take(256);
    w.fp_ss = take(static_cast<size_t>(d.M) * d.fp_groups * sizeof(float));
    w.gram = take(static_cast<size_t>(d.M) * d.S_max * sizeof(float));
    w.anchor = take(static_cast<size_t>(d.M) * sizeof(int32_t));
    const bool tok = d.B == 1;
    w.logits = take(tok ? 0 : static_cast<size_t>(d.M) * d.Hq * d.nb * sizeof(float));
    w.tok_split = take(tok ? static_cast<size_t>(3) * d.M * d.Hq * kHeadDim * 2 : 0);
    const int64_t ranges = tok ? (d.N + tok_range(d) - 1) / tok_range(d) : 0;
    w.tok_part = take(static_cast<size_t>(d.M) * d.Hq * ranges * 2 * sizeof(float));
    const size_t pack = tok ? static_cast<size_t>(d.M) * d.Hkv * tok_slots(d) * kHeadDim * 2 : 0;
    w.tok_list = take(tok ? static_cast<size_t>(d.M) * tok_slots(d) * sizeof(int32_t) : 0);
    w.tok_pack_k = take(pack);
    w.tok_pack_v = take(pack);
    w.tok_count = take(tok ? static_cast<size_t>(d.M) * sizeof(int32_t) : 0);
    w.topk_hist = take(tok ? static_cast<size_t>(d.M) * kTopkPasses * 256 * sizeof(int32_t) : 0);
    w.topk_state = take(tok ? static_cast<size_t>(d.M) * (kTopkPasses + 1) * 4 * sizeof(int32_t) : 0);
    w.topk_counts = take(tok ? static_cast<size_t>(d.M) * topk_max_chunks(d) * 2 * sizeof(int32_t) : 0);
    w.stats = take(static_cast<size_t>(d.M) * d.Hq * 2 * sizeof(float));
    w.scores = take(static_cast<size_t>(d.M) * d.nb * sizeof(float));
    w.total = off;
    return w;
}

namespace {

bool aligned(const void* ptr, size_t a) { return (reinterpret_cast<uintptr_t>(ptr) % a) == 0; }

// A device (or managed) allocation visible to the current device.
bool device_ptr(const void* ptr, size_t align)
{
    if (!ptr || !aligned(ptr, align)) return false;
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, ptr) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

int check_ws(const Derived& d, const void* ws, size_t ws_bytes)
{
    if (!device_ptr(ws, 256)) return SCALE_ERR_INVALID_ARG;
    if (ws_bytes < ws_layout(d).total) return SCALE_ERR_WORKSPACE;
    return SCALE_OK;
}

int check_range(const Derived& d, int mode, int64_t tb, int64_t te)
{
    if (mode != SCALE_MODE_PER_CLUSTER && mode != SCALE_MODE_PER_SUBCHUNK) return SCALE_ERR_INVALID_ARG;
    if (tb < 0 || te < tb || te > d.N) return SCALE_ERR_INVALID_ARG;
    const int64_t unit = mode == SCALE_MODE_PER_CLUSTER ? static_cast<int64_t>(d.per_outer) * d.L : d.L;
    if (tb % unit) return SCALE_ERR_INVALID_ARG;
    if (te != d.N && te % unit) return SCALE_ERR_INVALID_ARG;
    return SCALE_OK;
}

int cuda_status(cudaError_t e) { return e == cudaSuccess ? SCALE_OK : SCALE_ERR_CUDA; }

KvPaging contiguous(const Derived& d) { return KvPaging{nullptr, 0, 0, d.N, d.N}; }

// A page pool that the kernels can read: every box they load is 64 rows
// starting at a multiple of 64, so page sizes, sub-chunks, sinks, windows and
// blocks must be multiples of 64 (blocks may also be single tokens).
int check_pages(const Derived& d, const scale_kv_pages_t* kv, KvPaging* pg)
{
    if (!kv || kv->page_size <= 0 || kv->num_pages <= 0) return SCALE_ERR_INVALID_ARG;
    if (kv->page_size % 64 || d.L % 64 || d.n_sink % 64 || d.n_local % 64 || (d.B != 1 && d.B % 64))
        return SCALE_ERR_UNSUPPORTED;
    if (kv->num_pages * kv->page_size >= (1ll << 31) - 256) return SCALE_ERR_UNSUPPORTED;
    if (!device_ptr(kv->k_pages, 16) || !device_ptr(kv->v_pages, 16) || !device_ptr(kv->page_table, 4))
        return SCALE_ERR_INVALID_ARG;
    *pg = KvPaging{kv->page_table, kv->page_size, kv->num_pages, d.N, kv->num_pages * kv->page_size};
    return SCALE_OK;
}

struct Arena {
    size_t q, k, v, out, reps, fp, unit_start, n_units, sel, sel_count, ws, total;
};

Arena arena_layout(const Derived& d, int mode)
{
    (void)mode;
    Arena a{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t at = off;
        off = align_up(off + bytes, kAlign);
        return at;
    };
    a.q = take(static_cast<size_t>(d.N) * d.Hq * kHeadDim * 2);
    a.k = take(static_cast<size_t>(d.N) * d.Hkv * kHeadDim * 2);
    a.v = take(static_cast<size_t>(d.N) * d.Hkv * kHeadDim * 2);
    a.out = take(static_cast<size_t>(d.N) * d.Hq * kHeadDim * 2);
    a.reps = take(d.B == 1 ? 0 : static_cast<size_t>(d.Hkv) * d.nb * kHeadDim * sizeof(float));
    a.fp = take(static_cast<size_t>(d.M) * d.D * sizeof(float));
    a.unit_start = take(static_cast<size_t>(d.M + 1) * sizeof(int32_t));
    a.n_units = take(sizeof(int32_t));
    a.sel = take(static_cast<size_t>(d.M) * (d.k > 0 ? d.k : 1) * sizeof(int32_t));
    a.sel_count = take(static_cast<size_t>(d.M) * sizeof(int32_t));
    a.ws = take(ws_layout(d).total);
    a.total = off;
    return a;
}

// Two copy streams and the events of one scale_prefill_host call, released on
// every return.
struct CopyLanes {
    cudaStream_t in = nullptr, out = nullptr;
    std::vector<cudaEvent_t> events;
    cudaError_t event(cudaEvent_t* ev)
    {
        const cudaError_t e = cudaEventCreateWithFlags(ev, cudaEventDisableTiming);
        if (e == cudaSuccess) events.push_back(*ev);
        return e;
    }
    ~CopyLanes()
    {
        // an early error return leaves no copy running into the caller's buffers
        if (in) cudaStreamSynchronize(in);
        if (out) cudaStreamSynchronize(out);
        for (cudaEvent_t ev : events) cudaEventDestroy(ev);
        if (in) cudaStreamDestroy(in);
        if (out) cudaStreamDestroy(out);
    }
};

// Upper bound on the pieces of one scale_prefill_host call.
constexpr int kMaxHostPieces = 64;

}  // namespace
}  // namespace scale

using namespace scale;

extern "C" {

int scale_version(void) { return 10000; }

const char* scale_status_string(int s)
{
    switch (s) {
    case SCALE_OK: return "ok";
    case SCALE_ERR_INVALID_ARG: return "invalid argument";
    case SCALE_ERR_UNSUPPORTED: return "unsupported parameters";
    case SCALE_ERR_WORKSPACE: return "workspace too small";
    case SCALE_ERR_CUDA: return "CUDA runtime error";
    case SCALE_ERR_TIMEOUT: return "device wait timed out";
    case SCALE_ERR_DEVICE: return "device-side check failed";
    default: return "unknown status";
    }
}

int scale_workspace_size(const scale_params_t* p, int32_t mode, size_t* bytes)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    if (!bytes || (mode != SCALE_MODE_PER_CLUSTER && mode != SCALE_MODE_PER_SUBCHUNK))
        return SCALE_ERR_INVALID_ARG;
    *bytes = ws_layout(d).total;
    return SCALE_OK;
}

int scale_workspace_init(void* ws, size_t ws_bytes, scale_stream_t stream)
{
    if (!device_ptr(ws, 256) || ws_bytes < 256) return SCALE_ERR_INVALID_ARG;
    return cuda_status(cudaMemsetAsync(ws, 0, 256, stream));
}

// Outer chunks [*c_begin, *c_end) of the token range [tb, te): tb a multiple of
// the outer chunk length, te one too or N.
static int chunk_range(const Derived& d, int64_t tb, int64_t te, int* c_begin, int* c_end)
{
    const int64_t L_outer = static_cast<int64_t>(d.per_outer) * d.L;
    if (tb < 0 || te < tb || te > d.N || tb % L_outer || (te != d.N && te % L_outer))
        return SCALE_ERR_INVALID_ARG;
    *c_begin = static_cast<int>(tb / L_outer);
    *c_end = static_cast<int>((te + L_outer - 1) / L_outer);
    return SCALE_OK;
}

static int build_reps_impl(const Derived& d, int64_t tb, int64_t te, const void* q, const void* k,
                           const KvPaging& pg, float* reps, float* fingerprints, int32_t* unit_start,
                           int32_t* n_units, void* ws, size_t ws_bytes, scale_stream_t stream)
{
    int rc, c0, c1;
    if ((rc = chunk_range(d, tb, te, &c0, &c1))) return rc;
    if (!device_ptr(q, 16) || !device_ptr(k, 16) || !(device_ptr(reps, 16) || (!reps && d.B == 1)) ||
        !device_ptr(fingerprints, 16) || !device_ptr(unit_start, 4) || !device_ptr(n_units, 4))
        return SCALE_ERR_INVALID_ARG;
    if ((rc = check_ws(d, ws, ws_bytes))) return rc;
    return cuda_status(launch_build_reps_range(d, q, k, pg, reps, fingerprints, unit_start, n_units, c0,
                                               c1, static_cast<uint8_t*>(ws), stream));
}

int scale_build_reps(const scale_params_t* p, const void* q, const void* k, float* reps,
                     float* fingerprints, int32_t* unit_start, int32_t* n_units, void* ws,
                     size_t ws_bytes, scale_stream_t stream)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    return build_reps_impl(d, 0, d.N, q, k, contiguous(d), reps, fingerprints, unit_start, n_units, ws,
                           ws_bytes, stream);
}

int scale_build_reps_range(const scale_params_t* p, int64_t tok_begin, int64_t tok_end, const void* q,
                           const void* k, float* reps, float* fingerprints, int32_t* unit_start,
                           int32_t* n_units, void* ws, size_t ws_bytes, scale_stream_t stream)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    return build_reps_impl(d, tok_begin, tok_end, q, k, contiguous(d), reps, fingerprints, unit_start,
                           n_units, ws, ws_bytes, stream);
}

int scale_build_reps_paged(const scale_params_t* p, const void* q, const scale_kv_pages_t* kv, float* reps,
                           float* fingerprints, int32_t* unit_start, int32_t* n_units, void* ws,
                           size_t ws_bytes, scale_stream_t stream)
{
    Derived d;
    KvPaging pg;
    int rc = derive(p, &d);
    if (rc) return rc;
    if ((rc = check_pages(d, kv, &pg))) return rc;
    return build_reps_impl(d, 0, d.N, q, kv->k_pages, pg, reps, fingerprints, unit_start, n_units, ws,
                           ws_bytes, stream);
}

int scale_build_reps_range_paged(const scale_params_t* p, int64_t tok_begin, int64_t tok_end, const void* q,
                                 const scale_kv_pages_t* kv, float* reps, float* fingerprints,
                                 int32_t* unit_start, int32_t* n_units, void* ws, size_t ws_bytes,
                                 scale_stream_t stream)
{
    Derived d;
    KvPaging pg;
    int rc = derive(p, &d);
    if (rc) return rc;
    if ((rc = check_pages(d, kv, &pg))) return rc;
    return build_reps_impl(d, tok_begin, tok_end, q, kv->k_pages, pg, reps, fingerprints, unit_start,
                           n_units, ws, ws_bytes, stream);
}

int scale_select(const scale_params_t* p, int32_t mode, int64_t tok_begin, int64_t tok_end,
                 const float* reps, const float* fingerprints, const int32_t* unit_start,
                 const int32_t* n_units, int32_t* sel_blocks, int32_t* sel_count,
                 float* sel_scores, void* ws, size_t ws_bytes, scale_stream_t stream)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    if ((rc = check_range(d, mode, tok_begin, tok_end))) return rc;
    if (d.B == 1) return SCALE_ERR_UNSUPPORTED;  // block size 1: scale_select_tokens
    if (!device_ptr(reps, 16) || !device_ptr(fingerprints, 16) || !device_ptr(sel_count, 4) ||
        (d.k > 0 && !device_ptr(sel_blocks, 4)) || (sel_scores && !device_ptr(sel_scores, 4)))
        return SCALE_ERR_INVALID_ARG;
    if (mode == SCALE_MODE_PER_CLUSTER && (!device_ptr(unit_start, 4) || !device_ptr(n_units, 4)))
        return SCALE_ERR_INVALID_ARG;
    if ((rc = check_ws(d, ws, ws_bytes))) return rc;
    if (tok_begin == tok_end) return SCALE_OK;
    return cuda_status(launch_select(d, mode, tok_begin, tok_end, reps, fingerprints, unit_start,
                                     n_units, sel_blocks, sel_count, sel_scores,
                                     static_cast<uint8_t*>(ws), g_timeout_ns.load(), stream));
}

static int select_tokens_impl(const Derived& d, int32_t mode, int64_t tok_begin, int64_t tok_end,
                              const void* k, const KvPaging& pg, const float* fingerprints,
                              const int32_t* unit_start, const int32_t* n_units, int32_t* sel_tokens,
                              int32_t* sel_count, float* sel_scores, void* ws, size_t ws_bytes,
                              scale_stream_t stream)
{
    int rc;
    if (d.B != 1) return SCALE_ERR_INVALID_ARG;
    if (d.g > 8) return SCALE_ERR_UNSUPPORTED;  // token-level scoring: up to 8 query heads per KV head
    if ((rc = check_range(d, mode, tok_begin, tok_end))) return rc;
    if (!device_ptr(k, 16) || !device_ptr(fingerprints, 16) || !device_ptr(sel_count, 4) ||
        (d.k > 0 && !device_ptr(sel_tokens, 4)) || (sel_scores && !device_ptr(sel_scores, 4)))
        return SCALE_ERR_INVALID_ARG;
    if (mode == SCALE_MODE_PER_CLUSTER && (!device_ptr(unit_start, 4) || !device_ptr(n_units, 4)))
        return SCALE_ERR_INVALID_ARG;
    if ((rc = check_ws(d, ws, ws_bytes))) return rc;
    if (tok_begin == tok_end) return SCALE_OK;
    return cuda_status(launch_select_tokens(d, mode, tok_begin, tok_end, k, pg, fingerprints, unit_start,
                                            n_units, sel_tokens, sel_count, sel_scores,
                                            static_cast<uint8_t*>(ws), g_timeout_ns.load(), stream));
}

int scale_select_tokens(const scale_params_t* p, int32_t mode, int64_t tok_begin, int64_t tok_end,
                        const void* k, const float* fingerprints, const int32_t* unit_start,
                        const int32_t* n_units, int32_t* sel_tokens, int32_t* sel_count,
                        float* sel_scores, void* ws, size_t ws_bytes, scale_stream_t stream)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    return select_tokens_impl(d, mode, tok_begin, tok_end, k, contiguous(d), fingerprints, unit_start,
                              n_units, sel_tokens, sel_count, sel_scores, ws, ws_bytes, stream);
}

int scale_select_tokens_paged(const scale_params_t* p, int32_t mode, int64_t tok_begin, int64_t tok_end,
                              const scale_kv_pages_t* kv, const float* fingerprints,
                              const int32_t* unit_start, const int32_t* n_units, int32_t* sel_tokens,
                              int32_t* sel_count, float* sel_scores, void* ws, size_t ws_bytes,
                              scale_stream_t stream)
{
    Derived d;
    KvPaging pg;
    int rc = derive(p, &d);
    if (rc) return rc;
    if (d.B != 1) return SCALE_ERR_INVALID_ARG;
    if ((rc = check_pages(d, kv, &pg))) return rc;
    return select_tokens_impl(d, mode, tok_begin, tok_end, kv->k_pages, pg, fingerprints, unit_start,
                              n_units, sel_tokens, sel_count, sel_scores, ws, ws_bytes, stream);
}

static int sparse_prefill_impl(const Derived& d, int32_t mode, int64_t tok_begin, int64_t tok_end,
                               const void* q, const void* k, const void* v, const KvPaging& pg,
                               const int32_t* unit_start, const int32_t* n_units,
                               const int32_t* sel_blocks, const int32_t* sel_count, void* out, void* ws,
                               size_t ws_bytes, scale_stream_t stream)
{
    int rc;
    if ((rc = check_range(d, mode, tok_begin, tok_end))) return rc;
    if (d.B > 1 && max_distant_segments(d) > kMaxSegments) return SCALE_ERR_UNSUPPORTED;
    if (!device_ptr(q, 16) || !device_ptr(k, 16) || !device_ptr(v, 16) || !device_ptr(out, 16) ||
        !device_ptr(sel_count, 4) || (d.k > 0 && !device_ptr(sel_blocks, 4)))
        return SCALE_ERR_INVALID_ARG;
    if (mode == SCALE_MODE_PER_CLUSTER && (!device_ptr(unit_start, 4) || !device_ptr(n_units, 4)))
        return SCALE_ERR_INVALID_ARG;
    if ((rc = check_ws(d, ws, ws_bytes))) return rc;
    if (tok_begin == tok_end) return SCALE_OK;
    return cuda_status(launch_sparse_prefill(d, mode, tok_begin, tok_end, q, k, v, pg, unit_start,
                                             n_units, sel_blocks, sel_count, out,
                                             static_cast<uint8_t*>(ws), g_timeout_ns.load(), stream));
}

int scale_sparse_prefill(const scale_params_t* p, int32_t mode, int64_t tok_begin,
                         int64_t tok_end, const void* q, const void* k, const void* v,
                         const int32_t* unit_start, const int32_t* n_units,
                         const int32_t* sel_blocks, const int32_t* sel_count, void* out,
                         void* ws, size_t ws_bytes, scale_stream_t stream)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    return sparse_prefill_impl(d, mode, tok_begin, tok_end, q, k, v, contiguous(d), unit_start, n_units,
                               sel_blocks, sel_count, out, ws, ws_bytes, stream);
}

int scale_sparse_prefill_paged(const scale_params_t* p, int32_t mode, int64_t tok_begin, int64_t tok_end,
                               const void* q, const scale_kv_pages_t* kv, const int32_t* unit_start,
                               const int32_t* n_units, const int32_t* sel_blocks,
                               const int32_t* sel_count, void* out, void* ws, size_t ws_bytes,
                               scale_stream_t stream)
{
    Derived d;
    KvPaging pg;
    int rc = derive(p, &d);
    if (rc) return rc;
    if ((rc = check_pages(d, kv, &pg))) return rc;
    return sparse_prefill_impl(d, mode, tok_begin, tok_end, q, kv->k_pages, kv->v_pages, pg, unit_start,
                               n_units, sel_blocks, sel_count, out, ws, ws_bytes, stream);
}

int scale_get_device_status(const void* ws, scale_stream_t stream, int32_t* status)
{
    if (!device_ptr(ws, 256) || !status) return SCALE_ERR_INVALID_ARG;
    int32_t h = 0;
    cudaError_t e = cudaMemcpyAsync(&h, static_cast<const uint8_t*>(ws) + kStatusOffset, sizeof h,
                                    cudaMemcpyDeviceToHost, stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return SCALE_ERR_CUDA;
    *status = h;
    return SCALE_OK;
}

int scale_retrieval_calls(const scale_params_t* p, int32_t mode, const int32_t* unit_start_host,
                          int32_t n_units, int64_t* units, int64_t* calls)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    if (!units || !calls || (mode != SCALE_MODE_PER_CLUSTER && mode != SCALE_MODE_PER_SUBCHUNK))
        return SCALE_ERR_INVALID_ARG;
    const bool per_sub = mode == SCALE_MODE_PER_SUBCHUNK;
    if (!per_sub && (!unit_start_host || n_units < 0 || n_units > d.M)) return SCALE_ERR_INVALID_ARG;
    const int64_t n = per_sub ? d.M : n_units;
    int64_t c = 0;
    for (int64_t u = 0; u < n; ++u) {
        const int64_t a = per_sub ? u : unit_start_host[u];
        if (a < 0 || a >= d.M) return SCALE_ERR_INVALID_ARG;
        const int64_t s = a * d.L;
        const int64_t W = s - d.n_local > 0 ? s - d.n_local : 0;
        const int64_t lo = d.n_sink / d.B;
        int64_t hi = (W + d.B - 1) / d.B;
        if (hi > d.nb) hi = d.nb;
        if (hi > lo) ++c;
    }
    *units = n;
    *calls = c;
    return SCALE_OK;
}

int scale_prefill_host_arena_size(const scale_params_t* p, int32_t mode, size_t* bytes)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    if (!bytes || (mode != SCALE_MODE_PER_CLUSTER && mode != SCALE_MODE_PER_SUBCHUNK))
        return SCALE_ERR_INVALID_ARG;
    *bytes = arena_layout(d, mode).total;
    return SCALE_OK;
}

int scale_prefill_host(const scale_params_t* p, int32_t mode, const void* q_host,
                       const void* k_host, const void* v_host, void* out_host, void* arena,
                       size_t arena_bytes, scale_stream_t stream)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    if (mode != SCALE_MODE_PER_CLUSTER && mode != SCALE_MODE_PER_SUBCHUNK) return SCALE_ERR_INVALID_ARG;
    if (!q_host || !k_host || !v_host || !out_host || !device_ptr(arena, 256))
        return SCALE_ERR_INVALID_ARG;
    const Arena A = arena_layout(d, mode);
    if (arena_bytes < A.total) return SCALE_ERR_WORKSPACE;
    uint8_t* base = static_cast<uint8_t*>(arena);
    const size_t q_row = static_cast<size_t>(d.Hq) * kHeadDim * 2;
    const size_t kv_row_b = static_cast<size_t>(d.Hkv) * kHeadDim * 2;
    void* ws = base + A.ws;
    const size_t wsb = arena_bytes - A.ws;
    auto* reps = d.B == 1 ? nullptr : reinterpret_cast<float*>(base + A.reps);
    auto* fp = reinterpret_cast<float*>(base + A.fp);
    auto* us = reinterpret_cast<int32_t*>(base + A.unit_start);
    auto* nu = reinterpret_cast<int32_t*>(base + A.n_units);
    auto* sel = reinterpret_cast<int32_t*>(base + A.sel);
    auto* cnt = reinterpret_cast<int32_t*>(base + A.sel_count);

    // Pieces of whole outer chunks. Piece p computes once its own rows are on
    // the device (the rows before it arrived first, on the same copy stream);
    // its output rows go back while piece p + 1 computes. Every row a piece
    // reads lies before its end when L and n_local are multiples of 128 (the
    // causal window's 128-row tiles then end at the query block's end);
    // otherwise a tile may reach rows that the next piece's copy is writing,
    // and the call runs as one piece.
    const int n_chunks = outer_chunks(d);
    const bool split = d.L % 128 == 0 && d.n_local % 128 == 0;
    int per_piece = split ? (n_chunks + kMaxHostPieces - 1) / kMaxHostPieces : n_chunks;
    const int pieces = (n_chunks + per_piece - 1) / per_piece;
    const int64_t L_outer = static_cast<int64_t>(d.per_outer) * d.L;

    CopyLanes lanes;
    cudaEvent_t ev_start, ev_end;
    cudaError_t e = cudaStreamCreateWithFlags(&lanes.in, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&lanes.out, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = lanes.event(&ev_start);
    if (e == cudaSuccess) e = lanes.event(&ev_end);
    if (e == cudaSuccess) e = cudaEventRecord(ev_start, stream);  // the arena's earlier users
    if (e == cudaSuccess) e = cudaStreamWaitEvent(lanes.in, ev_start, 0);
    if (e != cudaSuccess) return SCALE_ERR_CUDA;
    if ((rc = scale_workspace_init(ws, wsb, stream))) return rc;

    for (int pc = 0; pc < pieces; ++pc) {
        const int64_t t0 = static_cast<int64_t>(pc) * per_piece * L_outer;
        const int64_t t1 = (pc + 1 == pieces) ? d.N : t0 + per_piece * L_outer;
        const size_t rows = static_cast<size_t>(t1 - t0);
        cudaEvent_t ev_in, ev_done;
        e = lanes.event(&ev_in);
        if (e == cudaSuccess) e = lanes.event(&ev_done);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(base + A.q + t0 * q_row, static_cast<const uint8_t*>(q_host) + t0 * q_row,
                                rows * q_row, cudaMemcpyHostToDevice, lanes.in);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(base + A.k + t0 * kv_row_b, static_cast<const uint8_t*>(k_host) + t0 * kv_row_b,
                                rows * kv_row_b, cudaMemcpyHostToDevice, lanes.in);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(base + A.v + t0 * kv_row_b, static_cast<const uint8_t*>(v_host) + t0 * kv_row_b,
                                rows * kv_row_b, cudaMemcpyHostToDevice, lanes.in);
        if (e == cudaSuccess) e = cudaEventRecord(ev_in, lanes.in);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(stream, ev_in, 0);
        if (e != cudaSuccess) return SCALE_ERR_CUDA;
        if ((rc = scale_build_reps_range(p, t0, t1, base + A.q, base + A.k, reps, fp, us, nu, ws, wsb, stream)))
            return rc;
        rc = d.B == 1 ? scale_select_tokens(p, mode, t0, t1, base + A.k, fp, us, nu, sel, cnt, nullptr, ws, wsb,
                                            stream)
                      : scale_select(p, mode, t0, t1, reps, fp, us, nu, sel, cnt, nullptr, ws, wsb, stream);
        if (rc) return rc;
        if ((rc = scale_sparse_prefill(p, mode, t0, t1, base + A.q, base + A.k, base + A.v, us, nu, sel, cnt,
                                       base + A.out, ws, wsb, stream)))
            return rc;
        e = cudaEventRecord(ev_done, stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(lanes.out, ev_done, 0);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(static_cast<uint8_t*>(out_host) + t0 * q_row, base + A.out + t0 * q_row,
                                rows * q_row, cudaMemcpyDeviceToHost, lanes.out);
        if (e != cudaSuccess) return SCALE_ERR_CUDA;
    }
    e = cudaEventRecord(ev_end, lanes.out);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(stream, ev_end, 0);
    if (e != cudaSuccess) return SCALE_ERR_CUDA;
    int32_t st = 0;
    if ((rc = scale_get_device_status(ws, stream, &st))) return rc;
    return st;
}

int scale_decode_cache_size(const scale_params_t* p, size_t* bytes)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    if (!bytes) return SCALE_ERR_INVALID_ARG;
    *bytes = align_up(decode_cache_bytes(d), kAlign);
    return SCALE_OK;
}

int scale_decode_cache_init(void* cache, size_t cache_bytes, scale_stream_t stream)
{
    if (!device_ptr(cache, 256) || cache_bytes < 256) return SCALE_ERR_INVALID_ARG;
    return cuda_status(cudaMemsetAsync(cache, 0, cache_bytes, stream));
}

int scale_decode_workspace_size(const scale_params_t* p, size_t* bytes)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    if (!bytes) return SCALE_ERR_INVALID_ARG;
    *bytes = decode_ws_bytes(d, decode_splits());
    return SCALE_OK;
}

int scale_decode_step(const scale_params_t* p, int64_t t, const void* q_t, const void* k, const void* v,
                      void* cache, size_t cache_bytes, void* out_t, void* ws, size_t ws_bytes,
                      scale_stream_t stream)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    if (d.B != 1) return SCALE_ERR_INVALID_ARG;
    if (d.g > 8 || d.Hq > 96) return SCALE_ERR_UNSUPPORTED;
    if (t < 0 || t >= d.N) return SCALE_ERR_INVALID_ARG;
    if (!device_ptr(q_t, 16) || !device_ptr(k, 16) || !device_ptr(v, 16) || !device_ptr(out_t, 16) ||
        !device_ptr(cache, 256) || !device_ptr(ws, 256))
        return SCALE_ERR_INVALID_ARG;
    if (cache_bytes < decode_cache_bytes(d) || ws_bytes < decode_ws_bytes(d, decode_splits()))
        return SCALE_ERR_WORKSPACE;
    return cuda_status(launch_decode_step(d, t, q_t, k, v, static_cast<uint8_t*>(cache), out_t,
                                          static_cast<uint8_t*>(ws), g_timeout_ns.load(), stream));
}

int scale_set_wait_timeout_ns(uint64_t ns)
{
    if (ns == 0) return SCALE_ERR_INVALID_ARG;
    g_timeout_ns.store(ns);
    return SCALE_OK;
}

int scale_selftest_wait_timeout(void* ws, size_t ws_bytes, uint64_t timeout_ns, scale_stream_t stream)
{
    if (!device_ptr(ws, 256) || ws_bytes < 256 || timeout_ns == 0) return SCALE_ERR_INVALID_ARG;
    return cuda_status(launch_wait_selftest(static_cast<uint8_t*>(ws), timeout_ns, stream));
}

}  // extern "C"
