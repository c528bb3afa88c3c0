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

// log2 of the partial slots a route's chunks use: 1 slot on the CUDA-core path. On the
// tensor-core path a work unit covers a group of 2^group_log2 routes in tiles of 128; a unit
// with n_a route tiles (rounded to 1, 2 or 4) splits each chunk over (group / 128) / n_a
// token-parity streams.
__device__ __forceinline__ int slots_log2(int M, int m, int sub_per_chunk, int group_log2) {
    if (sub_per_chunk == 1) return 0;
    const int ns_log2 = group_log2 - 7;
    const int g0 = (m >> group_log2) << group_log2;
    const int rem = M - g0;
    const int tiles = rem >= (1 << group_log2) ? (1 << ns_log2) : (rem + 127) >> 7;
    const int na_log2 = tiles <= 1 ? 0 : (tiles <= 2 ? 1 : 2);
    return ns_log2 - na_log2;
}

// Merge of the partial slots of one row (App. A.3):
//   g = max_r mx_r; w_r = 2^(mx_r - g); out = sum_r w_r acc_r / sum_r w_r l_r;
//   the row's base-2 log-normaliser is g + log2(sum_r w_r l_r).
// T = D / 4 channel groups per row (four channels each, one 16-byte load per slot), each taken
// by P adjacent lanes; a block of 256 threads covers 256 / (T P) rows of one (b, h), which
// blockIdx.y + gridDim.y * blockIdx.z names. The slots are taken KB at a time (all loads of a
// batch issued together): lane p of a group merges batches p, p + P, p + 2P, ... online, and
// the P partial merges are then combined by a butterfly over the group's lanes, whose result
// lane 0 writes. The order is fixed, so every run gives the same bits. P > 1 serves rows with
// many slots (many chunks of a group with one route tile, each in four token-parity parts),
// which one lane would take one batch after another.
template <int P>
__device__ __forceinline__ void merge_lanes(float& g, float& a, float4& u) {
    const unsigned lane = threadIdx.x & 31u;
    const unsigned mask = ((1u << P) - 1u) << (lane & ~(unsigned)(P - 1));
#pragma unroll
    for (int off = 1; off < P; off <<= 1) {
        const float g2 = __shfl_xor_sync(mask, g, off);
        const float a2 = __shfl_xor_sync(mask, a, off);
        const float x2 = __shfl_xor_sync(mask, u.x, off);
        const float y2 = __shfl_xor_sync(mask, u.y, off);
        const float z2 = __shfl_xor_sync(mask, u.z, off);
        const float w2 = __shfl_xor_sync(mask, u.w, off);
        const float gn = fmaxf(g, g2);
        if (gn == -INFINITY) continue;  // both halves empty so far
        const float s1 = fast_exp2(g - gn), s2 = fast_exp2(g2 - gn);  // 0 for an empty half
        a = a * s1 + a2 * s2;
        u.x = u.x * s1 + x2 * s2;
        u.y = u.y * s1 + y2 * s2;
        u.z = u.z * s1 + z2 * s2;
        u.w = u.w * s1 + w2 * s2;
        g = gn;
    }
}

template <int D, int KB, int P>
__global__ void __launch_bounds__(256)
    combine_kernel(const float* __restrict__ pmax, const float* __restrict__ psum,
                   const float* __restrict__ pacc, int64_t BH, int M, int nchunk,
                   int sub_per_chunk, int group_log2, float* __restrict__ out32,
                   __nv_bfloat16* __restrict__ outop, __nv_bfloat16* __restrict__ outlo,
                   float op_sign, float* __restrict__ lse) {
    constexpr int T = D / 4;
    constexpr int kRowsPerBlock = 256 / (T * P);
    static_assert(P == 1 || P == 2 || P == 4 || P == 8, "lanes per channel group");
    tc::pdl_trigger();
    tc::pdl_wait();  // the partials and the outputs belong to the kernels around this one
    const int64_t bh = (int64_t)blockIdx.z * gridDim.y + blockIdx.y;
    const int m = blockIdx.x * kRowsPerBlock + (int)(threadIdx.x / (T * P));
    const int q = (int)((threadIdx.x / P) % T);
    const int lp = (int)(threadIdx.x % P);
    // (all P lanes of a channel group share m, so they leave or stay together)
    if (bh >= BH || m >= M) return;
    const int ul = slots_log2(M, m, sub_per_chunk, group_log2);
    const int n = nchunk << ul;  // slot s: chunk s >> ul, part s & (2^ul - 1)
    const int64_t row = bh * M + m;
    // partial row of slot s: (bh * nchunk * sub + (s >> ul) * sub + (s & mask)) * M + m
    const int64_t base = bh * (int64_t)nchunk * sub_per_chunk * M + m;
    const int mask = (1 << ul) - 1;
    float g = -INFINITY, a = 0.f;
    float4 u = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s0 = lp * KB; s0 < n; s0 += KB * P) {
        float mx[KB], ps[KB];
        float4 v[KB];
#pragma unroll
        for (int j = 0; j < KB; ++j) {
            const int s = s0 + j;
            mx[j] = -INFINITY;
            ps[j] = 0.f;
            v[j] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (s < n) {
                const int64_t r =
                    base + ((int64_t)(s >> ul) * sub_per_chunk + (s & mask)) * (int64_t)M;
                mx[j] = __ldg(pmax + r);
                ps[j] = __ldg(psum + r);
                v[j] = __ldg(reinterpret_cast<const float4*>(pacc + r * D) + q);
            }
        }
        float gb = mx[0];
#pragma unroll
        for (int j = 1; j < KB; ++j) gb = fmaxf(gb, mx[j]);
        if (gb == -INFINITY) continue;  // every slot of the block is empty
        const float gn = fmaxf(g, gb);
        const float sc = fast_exp2(g - gn);  // 0 while g is -inf
        a *= sc;
        u.x *= sc;
        u.y *= sc;
        u.z *= sc;
        u.w *= sc;
#pragma unroll
        for (int j = 0; j < KB; ++j) {
            const float w = fast_exp2(mx[j] - gn);  // 0 for an empty slot
            a = fmaf(w, ps[j], a);
            u.x = fmaf(w, v[j].x, u.x);
            u.y = fmaf(w, v[j].y, u.y);
            u.z = fmaf(w, v[j].z, u.z);
            u.w = fmaf(w, v[j].w, u.w);
        }
        g = gn;
    }
    if constexpr (P > 1) {
        merge_lanes<P>(g, a, u);
        if (lp != 0) return;
    }
    const float inv = a > 0.f ? 1.f / a : 0.f;
    if (lse && q == 0) lse[row] = a > 0.f ? g + log2f(a) : -INFINITY;
    const float4 o = make_float4(u.x * inv, u.y * inv, u.z * inv, u.w * inv);
    reinterpret_cast<float4*>(out32 + row * D)[q] = o;
    if (outop) {
        const __nv_bfloat162 h01 = __floats2bfloat162_rn(op_sign * o.x, op_sign * o.y);
        const __nv_bfloat162 h23 = __floats2bfloat162_rn(op_sign * o.z, op_sign * o.w);
        uint2 pk;
        pk.x = *reinterpret_cast<const uint32_t*>(&h01);
        pk.y = *reinterpret_cast<const uint32_t*>(&h23);
        reinterpret_cast<uint2*>(outop + row * D)[q] = pk;
        if (outlo) {
            // what bf16 rounding left out: op_sign * o - hi, rounded to bf16 again
            const float2 h0 = __bfloat1622float2(h01), h1 = __bfloat1622float2(h23);
            const __nv_bfloat162 l0 =
                __floats2bfloat162_rn(op_sign * o.x - h0.x, op_sign * o.y - h0.y);
            const __nv_bfloat162 l1 =
                __floats2bfloat162_rn(op_sign * o.z - h1.x, op_sign * o.w - h1.y);
            uint2 pl;
            pl.x = *reinterpret_cast<const uint32_t*>(&l0);
            pl.y = *reinterpret_cast<const uint32_t*>(&l1);
            reinterpret_cast<uint2*>(outlo + row * D)[q] = pl;
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
                    float* lse, bool lo) {
    float* out32 = (float*)(ws + (call == 1 ? p.off_q32 : p.off_z32));
    __nv_bfloat16* outop = nullptr;
    if (p.path == kPathTc) outop = (__nv_bfloat16*)(ws + (call == 1 ? p.off_qop : p.off_zop));
    __nv_bfloat16* outlo = nullptr;
    if (lo && call == 1 && p.path == kPathTc) outlo = (__nv_bfloat16*)(ws + p.off_qlo);
    const float* pmax = (const float*)(ws + p.off_pmax);
    const float* psum = (const float*)(ws + p.off_psum);
    const float* pacc = (const float*)(ws + p.off_pacc);
    const float sign = negate ? -1.f : 1.f;
    // the group of routes a tensor-core unit covers is a power of two (tile rows x streams)
    int group_log2 = 0;
    if (p.sub_per_chunk > 1) {
        while ((int64_t(1) << group_log2) < p.tc_group) ++group_log2;
        if ((int64_t(1) << group_log2) != p.tc_group || group_log2 < 7) return cudaErrorInvalidValue;
    }
    if (p.nchunk * p.sub_per_chunk > INT32_MAX || p.M > INT32_MAX) return cudaErrorInvalidValue;
    // (b, h) over gridDim.y x gridDim.z (each at most 65535)
    const int64_t gy = p.BH < 65535 ? p.BH : 65535;
    const int64_t gz = (p.BH + gy - 1) / gy;
    if (gz > 65535) return cudaErrorInvalidValue;
    // slots per row at most: nchunk, times the token-parity parts of the last (partial) route
    // group's rows on the tensor-core path. Up to 32 slots (four batches), one lane per channel
    // group takes them; beyond that (many chunks of a one-tile group), four lanes share a row's
    // batches.
    int64_t n_slots = p.nchunk;
    if (p.sub_per_chunk > 1) {
        const int64_t group = int64_t(1) << group_log2, rem = p.M % group;
        const int64_t tiles = rem == 0 ? group / 128 : (rem + 127) / 128;
        const int64_t na = tiles <= 1 ? 1 : (tiles <= 2 ? 2 : 4);
        n_slots = p.nchunk * ((group / 128) / na);
    }
#define FLAREPP_COMBINE_P(DD, KB, PP)                                                         \
    {                                                                                         \
        constexpr int64_t rows = 256 / ((DD / 4) * PP);                                       \
        const int64_t gx = (p.M + rows - 1) / rows;                                           \
        return launch_pdl(combine_kernel<DD, KB, PP>,                                         \
                          dim3((unsigned)gx, (unsigned)gy, (unsigned)gz), dim3(256), 0, st,   \
                          pmax, psum, pacc, p.BH, (int)p.M, (int)p.nchunk,                    \
                          (int)p.sub_per_chunk, group_log2, out32, outop, outlo, sign, lse);  \
    }
#define FLAREPP_COMBINE(DD)                                   \
    {                                                         \
        if (n_slots <= 4) FLAREPP_COMBINE_P(DD, 4, 1)         \
        if (n_slots <= 32) FLAREPP_COMBINE_P(DD, 8, 1)        \
        FLAREPP_COMBINE_P(DD, 8, 4)                           \
    }
    switch (p.D) {
        case 16: FLAREPP_COMBINE(16)
        case 32: FLAREPP_COMBINE(32)
        case 64: FLAREPP_COMBINE(64)
    }
#undef FLAREPP_COMBINE
#undef FLAREPP_COMBINE_P
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
