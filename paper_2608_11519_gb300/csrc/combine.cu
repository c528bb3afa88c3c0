// Split-N combine shared by every path: the stable log-sum-exp merge of the chunk
// partials into Q (call 1) or Z (call 2), App. A.3.
#include <cuda_bf16.h>
#include <math.h>

#include "flarepp_internal.h"

namespace flarepp {
namespace {

__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// One warp per (bh, m): merge the chunk partials in ascending chunk order (App. A.3):
//   g = max_r mx_r; w_r = 2^(mx_r - g); out = sum_r w_r acc_r / sum_r w_r l_r.
template <int D>
__global__ void combine_kernel(const float* __restrict__ pmax, const float* __restrict__ psum,
                               const float* __restrict__ pacc, int64_t rows, int64_t M,
                               int64_t nchunk, float* __restrict__ out32,
                               __nv_bfloat16* __restrict__ outop) {
    constexpr int PER = (D + 31) / 32;
    const int lane = threadIdx.x & 31;
    const int64_t row = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
    if (row >= rows) return;
    const int64_t bh = row / M, m = row % M;
    float g = -INFINITY;
    for (int64_t c = 0; c < nchunk; ++c) g = fmaxf(g, pmax[(bh * nchunk + c) * M + m]);
    float a = 0.f, u[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) u[i] = 0.f;
    if (g != -INFINITY) {
        for (int64_t c = 0; c < nchunk; ++c) {
            const int64_t r = (bh * nchunk + c) * M + m;
            const float w = fast_exp2(pmax[r] - g);
            a = fmaf(w, psum[r], a);
#pragma unroll
            for (int i = 0; i < PER; ++i) {
                const int d = lane + 32 * i;
                if (d < D) u[i] = fmaf(w, pacc[r * D + d], u[i]);
            }
        }
    }
    const float inv = a > 0.f ? 1.f / a : 0.f;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const int d = lane + 32 * i;
        if (d < D) {
            const float val = u[i] * inv;
            out32[row * D + d] = val;
            if (outop) outop[row * D + d] = __float2bfloat16_rn(val);
        }
    }
}

}  // namespace

cudaError_t combine(const Plan& p, int call, char* ws, cudaStream_t st) {
    const int64_t rows = p.BH * p.M;
    const int warps = 8;
    const int64_t blocks = (rows + warps - 1) / warps;
    float* out32 = (float*)(ws + (call == 1 ? p.off_q32 : p.off_z32));
    __nv_bfloat16* outop = nullptr;
    if (p.path == kPathTc) outop = (__nv_bfloat16*)(ws + (call == 1 ? p.off_qop : p.off_zop));
    const float* pmax = (const float*)(ws + p.off_pmax);
    const float* psum = (const float*)(ws + p.off_psum);
    const float* pacc = (const float*)(ws + p.off_pacc);
    switch (p.D) {
        case 16:
            combine_kernel<16><<<(unsigned)blocks, warps * 32, 0, st>>>(pmax, psum, pacc, rows, p.M,
                                                                        p.nchunk, out32, outop);
            break;
        case 32:
            combine_kernel<32><<<(unsigned)blocks, warps * 32, 0, st>>>(pmax, psum, pacc, rows, p.M,
                                                                        p.nchunk, out32, outop);
            break;
        case 64:
            combine_kernel<64><<<(unsigned)blocks, warps * 32, 0, st>>>(pmax, psum, pacc, rows, p.M,
                                                                        p.nchunk, out32, outop);
            break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace flarepp
