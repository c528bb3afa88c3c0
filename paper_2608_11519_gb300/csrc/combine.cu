// Split-N combine shared by every path: the stable log-sum-exp merge of the chunk
// partials into Q (call 1) or Z (call 2), App. A.3.
#include <cuda_bf16.h>
#include <math.h>

#include "flarepp_internal.h"
#include "tc_ptx.cuh"

namespace flarepp {
namespace {

__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Partial slots a route's chunks use: 1 on the CUDA-core path. On the tensor-core path a
// work unit covers a group of `group` routes in tiles of 128; a unit with n_a route tiles
// (rounded to 1, 2 or 4) splits each chunk over (group / 128) / n_a token-parity streams.
__device__ __forceinline__ int slots_of_route(int64_t M, int64_t m, int64_t sub_per_chunk,
                                              int64_t group) {
    if (sub_per_chunk == 1) return 1;
    const int64_t ns = group / 128;
    const int64_t g = m / group;
    const int64_t rem = M - g * group;
    const int64_t tiles = rem >= group ? ns : (rem + 127) / 128;
    const int64_t na = tiles <= 1 ? 1 : (tiles <= 2 ? 2 : 4);
    return (int)(ns / na);
}

// One warp per (bh, m): merge the partial slots (App. A.3):
//   g = max_r mx_r; w_r = 2^(mx_r - g); out = sum_r w_r acc_r / sum_r w_r l_r;
//   the row's base-2 log-normaliser is g + log2(sum_r w_r l_r).
// The slots are taken KB (4 or 32) at a time, and every load of a block is issued at once:
// the lanes load one slot's maximum and sum each, and (lanes as channels) the values of all
// KB slots. The blocks are merged online with a running maximum, so a row costs one round of
// memory latency per KB slots (the merge is the same in every run: deterministic). KB = 4
// serves rows of at most four slots with few instructions.
template <int D, int KB>
__global__ void combine_kernel(const float* __restrict__ pmax, const float* __restrict__ psum,
                               const float* __restrict__ pacc, int64_t rows, int64_t M,
                               int64_t nchunk, int64_t sub_per_chunk, int64_t group,
                               float* __restrict__ out32,
                               __nv_bfloat16* __restrict__ outop, float op_sign,
                               float* __restrict__ lse) {
    constexpr int PER = (D + 31) / 32;
    tc::pdl_trigger();
    tc::pdl_wait();  // the partials and the outputs belong to the kernels around this one
    const int lane = threadIdx.x & 31;
    const int64_t row = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
    if (row >= rows) return;
    const int64_t bh = row / M, m = row % M;
    const int used = slots_of_route(M, m, sub_per_chunk, group);
    const int64_t nslot = nchunk * sub_per_chunk;
    const int64_t n = nchunk * used;  // the row's slots, s -> chunk s / used, part s % used
    auto slot_row = [&](int64_t s) {
        return (bh * nslot + (s / used) * sub_per_chunk + s % used) * M + m;
    };
    float g = -INFINITY, a = 0.f, u[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) u[i] = 0.f;
    for (int64_t s0 = 0; s0 < n; s0 += KB) {
        const int cnt = (int)min((int64_t)KB, n - s0);
        const bool in = lane < cnt;
        const int64_t rl = in ? slot_row(s0 + lane) : 0;
        const float mx = in ? pmax[rl] : -INFINITY;
        const float ps = in ? psum[rl] : 0.f;
        float v[KB][PER];
#pragma unroll
        for (int j = 0; j < KB; ++j) {
            const int64_t rj = j < cnt ? slot_row(s0 + j) : 0;
#pragma unroll
            for (int i = 0; i < PER; ++i) {
                const int d = lane + 32 * i;
                v[j][i] = (j < cnt && d < D) ? pacc[rj * D + d] : 0.f;
            }
        }
        float gb = mx;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) gb = fmaxf(gb, __shfl_xor_sync(0xffffffffu, gb, off));
        if (gb == -INFINITY) continue;  // every slot of the block is empty
        const float gn = fmaxf(g, gb);
        const float sc = fast_exp2(g - gn);  // 0 while g is -inf
        a *= sc;
#pragma unroll
        for (int i = 0; i < PER; ++i) u[i] *= sc;
        const float w = in ? fast_exp2(mx - gn) : 0.f;
        float aw = w * ps;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) aw += __shfl_xor_sync(0xffffffffu, aw, off);
        a += aw;
#pragma unroll
        for (int j = 0; j < KB; ++j) {
            const float wj = __shfl_sync(0xffffffffu, w, j);
#pragma unroll
            for (int i = 0; i < PER; ++i) u[i] = fmaf(wj, v[j][i], u[i]);
        }
        g = gn;
    }
    const float inv = a > 0.f ? 1.f / a : 0.f;
    if (lse && lane == 0) lse[row] = a > 0.f ? g + log2f(a) : -INFINITY;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const int d = lane + 32 * i;
        if (d < D) {
            const float val = u[i] * inv;
            out32[row * D + d] = val;
            if (outop) outop[row * D + d] = __float2bfloat16_rn(op_sign * val);
        }
    }
}

__global__ void negate_bf16_kernel(const __nv_bfloat16* __restrict__ src,
                                   __nv_bfloat16* __restrict__ dst, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = __hneg(src[i]);
}

}  // namespace

cudaError_t combine(const Plan& p, int call, char* ws, bool negate, cudaStream_t st,
                    float* lse) {
    const int64_t rows = p.BH * p.M;
    const int warps = 8;
    const int64_t blocks = (rows + warps - 1) / warps;
    float* out32 = (float*)(ws + (call == 1 ? p.off_q32 : p.off_z32));
    __nv_bfloat16* outop = nullptr;
    if (p.path == kPathTc) outop = (__nv_bfloat16*)(ws + (call == 1 ? p.off_qop : p.off_zop));
    const float* pmax = (const float*)(ws + p.off_pmax);
    const float* psum = (const float*)(ws + p.off_psum);
    const float* pacc = (const float*)(ws + p.off_pacc);
    const float sign = negate ? -1.f : 1.f;
    // slots per row at most: nchunk x sub_per_chunk
    const bool few = p.nchunk * p.sub_per_chunk <= 4;
#define FLAREPP_COMBINE(DD)                                                                    \
    return launch_pdl(few ? combine_kernel<DD, 4> : combine_kernel<DD, 32>,                   \
                      dim3((unsigned)blocks), dim3(warps * 32), 0, st, pmax, psum, pacc, rows, \
                      p.M, p.nchunk, p.sub_per_chunk, p.tc_group, out32, outop, sign, lse);
    switch (p.D) {
        case 16: FLAREPP_COMBINE(16)
        case 32: FLAREPP_COMBINE(32)
        case 64: FLAREPP_COMBINE(64)
    }
#undef FLAREPP_COMBINE
    return cudaErrorInvalidValue;
}

cudaError_t negate_bf16(const void* src, void* dst, int64_t n, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    const int64_t blocks = (n + 255) / 256 < 1024 ? (n + 255) / 256 : 1024;
    negate_bf16_kernel<<<(unsigned)blocks, 256, 0, st>>>((const __nv_bfloat16*)src,
                                                         (__nv_bfloat16*)dst, n);
    return cudaGetLastError();
}

}  // namespace flarepp
