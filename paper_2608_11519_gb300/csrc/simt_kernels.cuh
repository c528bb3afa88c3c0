// CUDA-core kernels of the routing chain: the float32 dtype path (instantiated in
// simt_f32.cu). Products and accumulation in float32; tf32 tensor cores could not meet
// the float32 tolerance.
//
// Encode (calls 1 and 2, Sec. 3.2): one thread per route row streams a chunk of tokens
// through an online softmax (running max, running sum, weighted value sum) and writes
// the chunk's partials. Combine merges the partials of all chunks by the stable
// log-sum-exp reduction of App. A.3. Decode (call 3): one thread per token streams the M
// routes through an online softmax over routes.
//
// Scores are kept in the base-2 domain: x = (scale * log2 e) <q, k>, weights 2^(x - max).
#include <cuda_bf16.h>
#include <math.h>

#include "flarepp_internal.h"

#pragma once
#include <cuda_runtime.h>

namespace flarepp {
namespace simt {

constexpr float kLog2e = 1.4426950408889634f;
constexpr int kTile = 16;  // tokens (encode) or routes (decode) staged per step

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }
__device__ __forceinline__ void from_f32(float* p, float x) { *p = x; }
__device__ __forceinline__ void from_f32(__nv_bfloat16* p, float x) { *p = __float2bfloat16_rn(x); }

__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// grid.x = nchunk * n_mtiles * BH; block = m_tile threads.
template <int D, typename T, typename QT>
__global__ void __launch_bounds__(128) simt_encode_kernel(
    const T* __restrict__ k, const T* __restrict__ v, const QT* __restrict__ q, int q_per_head,
    int64_t H, int64_t N, int64_t M, int64_t chunk_len, int64_t nchunk, int64_t n_mtiles,
    float sl2, float* __restrict__ pmax, float* __restrict__ psum, float* __restrict__ pacc) {
    __shared__ float ks[kTile][D];
    __shared__ float vs[kTile][D];

    int64_t bid = blockIdx.x;
    const int64_t c = bid % nchunk;
    bid /= nchunk;
    const int64_t mt = bid % n_mtiles;
    const int64_t bh = bid / n_mtiles;
    const int64_t m = mt * blockDim.x + threadIdx.x;
    const bool active = m < M;

    // query row, pre-scaled into the base-2 domain
    float qr[D];
    {
        const int64_t qrow = (q_per_head ? (bh % H) : bh) * M + (active ? m : 0);
        const QT* qp = q + qrow * D;
#pragma unroll
        for (int d = 0; d < D; ++d) qr[d] = active ? to_f32(qp[d]) * sl2 : 0.f;
    }
    float o[D];
#pragma unroll
    for (int d = 0; d < D; ++d) o[d] = 0.f;
    float mx = -INFINITY, l = 0.f;

    const int64_t n_begin = c * chunk_len;
    const int64_t n_end = min(N, n_begin + chunk_len);
    const T* kb = k + bh * N * D;
    const T* vb = v + bh * N * D;
    for (int64_t n0 = n_begin; n0 < n_end; n0 += kTile) {
        const int cnt = (int)min((int64_t)kTile, n_end - n0);
        __syncthreads();
        for (int i = threadIdx.x; i < kTile * D; i += blockDim.x) {
            const int j = i / D, d = i % D;
            const bool in = j < cnt;
            ks[j][d] = in ? to_f32(kb[(n0 + j) * D + d]) : 0.f;
            vs[j][d] = in ? to_f32(vb[(n0 + j) * D + d]) : 0.f;
        }
        __syncthreads();
        float sc[kTile];
        float tmax = -INFINITY;
#pragma unroll
        for (int j = 0; j < kTile; ++j) {
            float acc = 0.f;
#pragma unroll
            for (int d = 0; d < D; ++d) acc = fmaf(qr[d], ks[j][d], acc);
            sc[j] = j < cnt ? acc : -INFINITY;
            tmax = fmaxf(tmax, sc[j]);
        }
        const float mnew = fmaxf(mx, tmax);
        const float corr = fast_exp2(mx - mnew);  // 0 on the first tile
        l *= corr;
#pragma unroll
        for (int d = 0; d < D; ++d) o[d] *= corr;
#pragma unroll
        for (int j = 0; j < kTile; ++j) {
            const float pj = fast_exp2(sc[j] - mnew);  // 0 for masked tokens
            l += pj;
#pragma unroll
            for (int d = 0; d < D; ++d) o[d] = fmaf(pj, vs[j][d], o[d]);
        }
        mx = mnew;
    }
    if (active) {
        const int64_t row = (bh * nchunk + c) * M + m;
        pmax[row] = mx;
        psum[row] = l;
#pragma unroll
        for (int d = 0; d < D; ++d) pacc[row * D + d] = o[d];
    }
}

// grid.x = ceil(N / 128) * BH; one thread per token; routes staged kTile at a time.
template <int D, typename T>
__global__ void __launch_bounds__(128) simt_decode_kernel(
    const T* __restrict__ k, const float* __restrict__ q32, const float* __restrict__ z32,
    int64_t N, int64_t M, float sl2, T* __restrict__ y, float* __restrict__ lse) {
    __shared__ float qs[kTile][D];
    __shared__ float zs[kTile][D];
    const int64_t ntiles = (N + 127) / 128;
    const int64_t bh = blockIdx.x / ntiles;
    const int64_t n = (blockIdx.x % ntiles) * 128 + threadIdx.x;
    const bool active = n < N;
    float kr[D], o[D];
    const T* kp = k + (bh * N + (active ? n : 0)) * D;
#pragma unroll
    for (int d = 0; d < D; ++d) {
        kr[d] = active ? to_f32(kp[d]) * sl2 : 0.f;
        o[d] = 0.f;
    }
    float mx = -INFINITY, l = 0.f;
    const float* qb = q32 + bh * M * D;
    const float* zb = z32 + bh * M * D;
    for (int64_t m0 = 0; m0 < M; m0 += kTile) {
        const int cnt = (int)min((int64_t)kTile, M - m0);
        __syncthreads();
        for (int i = threadIdx.x; i < kTile * D; i += blockDim.x) {
            const int j = i / D, d = i % D;
            const bool in = j < cnt;
            qs[j][d] = in ? qb[(m0 + j) * D + d] : 0.f;
            zs[j][d] = in ? zb[(m0 + j) * D + d] : 0.f;
        }
        __syncthreads();
        float sc[kTile];
        float tmax = -INFINITY;
#pragma unroll
        for (int j = 0; j < kTile; ++j) {
            float acc = 0.f;
#pragma unroll
            for (int d = 0; d < D; ++d) acc = fmaf(kr[d], qs[j][d], acc);
            sc[j] = j < cnt ? acc : -INFINITY;
            tmax = fmaxf(tmax, sc[j]);
        }
        const float mnew = fmaxf(mx, tmax);
        const float corr = fast_exp2(mx - mnew);
        l *= corr;
#pragma unroll
        for (int d = 0; d < D; ++d) o[d] *= corr;
#pragma unroll
        for (int j = 0; j < kTile; ++j) {
            const float pj = fast_exp2(sc[j] - mnew);
            l += pj;
#pragma unroll
            for (int d = 0; d < D; ++d) o[d] = fmaf(pj, zs[j][d], o[d]);
        }
        mx = mnew;
    }
    if (active) {
        const float inv = 1.f / l;
        T* yp = y + (bh * N + n) * D;
#pragma unroll
        for (int d = 0; d < D; ++d) from_f32(yp + d, o[d] * inv);
        if (lse) lse[bh * N + n] = mx + log2f(l);
    }
}

template <typename T>
cudaError_t encode_t(const Plan& p, int call, const void* k, const void* v, const void* seeds,
                     float scale, char* ws, cudaStream_t st) {
    const int64_t blocks = p.nchunk * p.n_mtiles * p.BH;
    const int threads = (int)p.m_tile;
    const float sl2 = scale * kLog2e;
    float* pmax = (float*)(ws + p.off_pmax);
    float* psum = (float*)(ws + p.off_psum);
    float* pacc = (float*)(ws + p.off_pacc);
    const T* kk = (const T*)k;
    const T* vv = (const T*)v;
#define FLAREPP_ENC(DD)                                                                         \
    if (call == 1)                                                                              \
        simt_encode_kernel<DD, T, T><<<(unsigned)blocks, threads, 0, st>>>(                     \
            kk, vv, (const T*)seeds, 1, p.H, p.N, p.M, p.chunk_len, p.nchunk, p.n_mtiles, sl2, \
            pmax, psum, pacc);                                                                  \
    else                                                                                        \
        simt_encode_kernel<DD, T, float><<<(unsigned)blocks, threads, 0, st>>>(                 \
            kk, vv, (const float*)(ws + p.off_q32), 0, p.H, p.N, p.M, p.chunk_len, p.nchunk,   \
            p.n_mtiles, sl2, pmax, psum, pacc);
    switch (p.D) {
        case 16: FLAREPP_ENC(16) break;
        case 32: FLAREPP_ENC(32) break;
        case 64: FLAREPP_ENC(64) break;
        default: return cudaErrorInvalidValue;
    }
#undef FLAREPP_ENC
    return cudaGetLastError();
}

template <typename T>
cudaError_t decode_t(const Plan& p, const void* K, float scale, void* Y, char* ws,
                     cudaStream_t st, float* lse) {
    const int64_t blocks = ((p.N + 127) / 128) * p.BH;
    const float sl2 = scale * kLog2e;
    const float* q32 = (const float*)(ws + p.off_q32);
    const float* z32 = (const float*)(ws + p.off_z32);
    switch (p.D) {
        case 16:
            simt_decode_kernel<16, T><<<(unsigned)blocks, 128, 0, st>>>((const T*)K, q32, z32, p.N,
                                                                         p.M, sl2, (T*)Y, lse);
            break;
        case 32:
            simt_decode_kernel<32, T><<<(unsigned)blocks, 128, 0, st>>>((const T*)K, q32, z32, p.N,
                                                                         p.M, sl2, (T*)Y, lse);
            break;
        case 64:
            simt_decode_kernel<64, T><<<(unsigned)blocks, 128, 0, st>>>((const T*)K, q32, z32, p.N,
                                                                         p.M, sl2, (T*)Y, lse);
            break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace simt
}  // namespace flarepp
