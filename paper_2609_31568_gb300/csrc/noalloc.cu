// noalloc.cu -- scale_build_reps_noalloc: step (a) for callers that cannot
// provide a workspace.
//
// Some callers cannot allocate device memory for us: a host framework's
// plugin interface that hands over only the input and output buffers, or a
// serving loop whose memory pool is fully reserved up front and where a
// cudaMalloc (which may synchronise the device) is not allowed on the request
// path. For them this entry point keeps step (a)'s scratch (the sums of
// squares of the fingerprints' column groups, the banded cosine matrix and
// the anchor flags) in the
// fixed array below, which every GPU that loads the library holds until the
// process exits. The kernels and their launch are the ones of
// scale_build_reps; only the scratch location differs.
#include <mutex>

#include "scale_internal.h"

namespace scale {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;  // 16 MiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) uint8_t g_scratch[kNoAllocScratchBytes];

std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_scratch on the current device, looked up once per device.
int scratch_address(void** out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SCALE_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_addr[dev]) {
        void* ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_scratch) != cudaSuccess || !ptr) {
            cudaGetLastError();
            return SCALE_ERR_CUDA;
        }
        g_scratch_addr[dev] = ptr;
    }
    *out = g_scratch_addr[dev];
    return SCALE_OK;
}

bool dev_ptr(const void* ptr, size_t align)
{
    if (!ptr || reinterpret_cast<uintptr_t>(ptr) % align) return false;
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, ptr) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

}  // namespace
}  // namespace scale

using namespace scale;

extern "C" int scale_build_reps_noalloc(const scale_params_t* p, const void* q, const void* k,
                                        float* reps, float* fingerprints, int32_t* unit_start,
                                        int32_t* n_units, scale_stream_t stream)
{
    Derived d;
    int rc = derive(p, &d);
    if (rc) return rc;
    if (!dev_ptr(q, 16) || !dev_ptr(k, 16) || !(dev_ptr(reps, 16) || (!reps && d.B == 1)) ||
        !dev_ptr(fingerprints, 16) ||
        !dev_ptr(unit_start, 4) || !dev_ptr(n_units, 4))
        return SCALE_ERR_INVALID_ARG;
    // Step (a) uses the workspace prefix that ends where the selection's regions begin.
    const size_t need = ws_layout(d).logits;
    if (need > kNoAllocScratchBytes) return SCALE_ERR_WORKSPACE;
    void* scratch = nullptr;
    if ((rc = scratch_address(&scratch))) return rc;
    // The array keeps the previous call's contents. Step (a) writes every
    // scratch element before reading it, so nothing needs clearing; its
    // kernels record no device status (they have no bounded waits and no
    // device-side checks), so the status word at the array's start is never
    // written or read.
    const KvPaging pg{nullptr, 0, 0, d.N, d.N};
    return launch_build_reps(d, q, k, pg, reps, fingerprints, unit_start, n_units,
                             static_cast<uint8_t*>(scratch), stream) == cudaSuccess
               ? SCALE_OK
               : SCALE_ERR_CUDA;
}
