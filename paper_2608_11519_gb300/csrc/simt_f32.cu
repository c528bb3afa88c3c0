// Instantiation of the CUDA-core encode and decode for f32 inputs.
#include "simt_kernels.cuh"

namespace flarepp {

cudaError_t simt_encode_f32(const Plan& p, int call, const void* k, const void* v,
                          const void* seeds, float scale, char* ws, cudaStream_t st) {
    return simt::encode_t<float>(p, call, k, v, seeds, scale, ws, st);
}

cudaError_t simt_decode_f32(const Plan& p, const void* K, float scale, void* Y, char* ws,
                          cudaStream_t st, float* lse) {
    return simt::decode_t<float>(p, K, scale, Y, ws, st, lse);
}

}  // namespace flarepp
