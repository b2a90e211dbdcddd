// tma_host.h -- host-side construction of TMA tensor maps for the token-major
// bf16 tensors the library reads ([tokens][heads][head_dim], head_dim innermost).
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <cstdint>

namespace scale_host {

// cuTensorMapEncodeTiled, resolved once through the runtime's driver entry point
// so that the library needs no link-time dependency on libcuda.
inline PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

// A 3-D map over bf16 [n_tokens][n_heads][head_dim] with a box of
// box_d x 1 x box_t elements and 128-byte swizzle (box_d * 2 must be <= 128).
// Out-of-range rows are filled with zeros. Returns false on failure.
inline bool make_token_major_map(CUtensorMap* map, const void* base, uint64_t head_dim,
                                 uint64_t n_heads, uint64_t n_tokens, uint32_t box_d,
                                 uint32_t box_t)
{
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    const cuuint64_t dims[3] = {head_dim, n_heads, n_tokens};
    const cuuint64_t strides[2] = {head_dim * 2, head_dim * n_heads * 2};
    const cuuint32_t box[3] = {box_d, 1, box_t};
    const cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                     strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// A map over a dense bf16 tensor of `rank` dimensions (dims[0] innermost,
// 128 elements of 2 bytes = 256-byte rows), with 128-byte swizzle and the
// given box. Returns false on failure.
inline bool make_dense_bf16_map(CUtensorMap* map, const void* base, uint32_t rank,
                                const uint64_t* dims, const uint32_t* box)
{
    auto enc = tensor_map_encoder();
    if (!enc || rank < 1 || rank > 5) return false;
    cuuint64_t d[5], str[4];
    cuuint32_t b[5], e[5];
    uint64_t stride = 2;
    for (uint32_t i = 0; i < rank; ++i) {
        d[i] = dims[i];
        b[i] = box[i];
        e[i] = 1;
        stride *= dims[i];
        if (i + 1 < rank) str[i] = stride;
    }
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), d, str, b,
                     e, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

}  // namespace scale_host
