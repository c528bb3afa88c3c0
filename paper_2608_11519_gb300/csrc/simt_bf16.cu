// Instantiation of the CUDA-core encode and decode for bf16 inputs.
#include "simt_kernels.cuh"

namespace flarepp {

cudaError_t simt_encode_bf16(const Plan& p, int call, const void* k, const void* v,
                          const void* seeds, float scale, char* ws, cudaStream_t st) {
    return simt::encode_t<__nv_bfloat16>(p, call, k, v, seeds, scale, ws, st);
}

cudaError_t simt_decode_bf16(const Plan& p, const void* K, float scale, void* Y, char* ws,
                          cudaStream_t st) {
    return simt::decode_t<__nv_bfloat16>(p, K, scale, Y, ws, st);
}

}  // namespace flarepp
