// Backward of the routing chain (App. A.5): the CUDA-core passes (float32 inputs), the
// kernels both paths share (c of call 3, the reduces of the route passes' partials) and
// the launch sequence of both paths; the tensor-core passes are in tc_bwd.cu.
//
// Every SDPA of the chain is differentiated from its saved output O and log-normaliser L:
//   P = 2^(x - L) with x = scale * log2(e) <a, b> (L kept in base 2 by the forward),
//   c = <dO, O>_D,  dS = P o (dO C^T - c),  dA = s dS B,  dB = s dS^T A,  dC = P^T dO
// for SDPA(A, B, C) with output O. The chain runs the three calls backwards:
//   call 3  Y = SDPA(K, Q, Z):   c3 per token;  dZ = P3^T dY,  dQ += s dS3^T K,  dK += s dS3 Q
//   call 2  Z = SDPA(Q, K, V):   c2 per route;  dV = P2^T dZ,  dQ += s dS2 K,    dK += s dS2^T Q
//   call 1  Q = SDPA(Qs, Kt, Vt) with the summed dQ (App. A.5: the decoder's query gradient is
//           added to the encoder's): c1 per route; dVt = P1^T dQ, dKt = s dS1^T Qs,
//           dQs = s dS1 Kt, summed over the batch for the shared seeds.
//
// Two kernel shapes cover it on CUDA cores. A route pass gives one thread per route and
// streams a chunk of tokens, accumulating the latent-side sums (dZ, dQ, dQs) into per-chunk
// partials that a reduce kernel adds in chunk order. A token pass gives one thread per
// token and streams every route, producing that token's dK, dV (calls 2 and 3 together) or
// dKt, dVt (call 1). The tensor-core path has the same structure (passes R3, T23, R2, T1,
// R1) with bf16 copies of Q, Z, dZ and dQ as MMA operands.
#include <cuda_bf16.h>
#include <math.h>

#include "flarepp_internal.h"

namespace flarepp {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr int kTok = 16;    // tokens staged per step of a route pass
constexpr int kRoute = 16;  // routes staged per step of a token pass

__device__ __forceinline__ float ld_f32(const float* p) { return *p; }
__device__ __forceinline__ float ld_f32(const __nv_bfloat16* p) { return __bfloat162float(*p); }
__device__ __forceinline__ void st_out(float* p, float x) { *p = x; }
__device__ __forceinline__ void st_out(__nv_bfloat16* p, float x) { *p = __float2bfloat16_rn(x); }

// The bf16 forward multiplies bf16 copies of Q and Z (its MMA operands); the backward
// differentiates that same function, so on the bf16 path it rounds Q and Z alike wherever
// they enter a product (logits, and Z in call 3's values).
template <typename T>
__device__ __forceinline__ float operand(float x) {
    if constexpr (sizeof(T) == 2) return __bfloat162float(__float2bfloat16_rn(x));
    return x;
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// c3[n] = <dY_n, Y_n>: each thread reads one 16-byte vector of a row of dY and of Y (so a
// warp reads consecutive rows whole), and the D / V threads of a row add their partial dot
// products with shuffles. rows * D / V threads in all.
template <int D, typename T>
__global__ void __launch_bounds__(256) delta_tokens_kernel(const T* __restrict__ dY,
                                                           const T* __restrict__ Y, int64_t rows,
                                                           float* __restrict__ c3) {
    constexpr int V = 16 / (int)sizeof(T);  // elements per 16-byte vector
    constexpr int TPR = D / V;              // threads per row (2 .. 16, a power of two)
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t r = t / TPR;
    float acc = 0.f;
    if (r < rows) {
        const uint4 a = reinterpret_cast<const uint4*>(dY)[t];
        const uint4 b = reinterpret_cast<const uint4*>(Y)[t];
        const T* av = reinterpret_cast<const T*>(&a);
        const T* bv = reinterpret_cast<const T*>(&b);
#pragma unroll
        for (int e = 0; e < V; ++e) acc = fmaf(ld_f32(av + e), ld_f32(bv + e), acc);
    }
#pragma unroll
    for (int off = TPR / 2; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (r < rows && (t % TPR) == 0) c3[r] = acc;
}

template <int D, typename T>
void launch_delta_tokens(const T* dY, const T* Y, int64_t rows, float* c3, cudaStream_t st) {
    constexpr int TPR = D / (16 / (int)sizeof(T));
    const int64_t threads = rows * TPR;
    delta_tokens_kernel<D, T><<<(unsigned)((threads + 255) / 256), 256, 0, st>>>(dY, Y, rows, c3);
}

// bf16 copy of a float32 array (the tensor-core passes' Q and Z operands)
__global__ void to_bf16_kernel(const float* __restrict__ src, __nv_bfloat16* __restrict__ dst,
                               int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = __float2bfloat16_rn(src[i]);
}

// hi = bf16(src), lo = bf16(src - hi): the operand pair the training forward gave Q
__global__ void to_bf16_hilo_kernel(const float* __restrict__ src, __nv_bfloat16* __restrict__ hi,
                                    __nv_bfloat16* __restrict__ lo, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const __nv_bfloat16 h = __float2bfloat16_rn(src[i]);
        hi[i] = h;
        lo[i] = __float2bfloat16_rn(src[i] - __bfloat162float(h));
    }
}

// Route pass of call MODE (3, 2 or 1) over one chunk of tokens; thread = route m.
//   MODE 3: a = Q, keys b = K, w = dY, g = Z, column statistics L3[n], c3[n];
//           pa += P w (dZ), pb += dS k (dQ / s)
//   MODE 2: a = Q, keys = K, w = V, g = dZ, row statistics L2[m], c2[m]; pb += dS k
//   MODE 1: a = seeds (per head), keys = Kt, w = Vt, g = dQ, row statistics L1[m], c1[m];
//           pb += dS kt
// dS here is P o (dP - c); the factor s is applied by the reduce.
// grid.x = nchunk * n_mtiles * BH; block = m_tile threads.
template <int D, typename T, typename AT, int MODE>
__global__ void __launch_bounds__(128) route_pass_kernel(
    const AT* __restrict__ a, int a_per_head, const T* __restrict__ kb, const T* __restrict__ wb,
    const float* __restrict__ g, const float* __restrict__ Lrow, const float* __restrict__ crow,
    const float* __restrict__ Lcol, const float* __restrict__ ccol, int64_t H, int64_t N,
    int64_t M, int64_t chunk_len, int64_t nchunk, int64_t n_mtiles, float sl2,
    float* __restrict__ pa, float* __restrict__ pb) {
    __shared__ float ks[kTok][D];
    __shared__ float ws[kTok][D];
    __shared__ float lc[kTok], cc[kTok];

    int64_t bid = blockIdx.x;
    const int64_t c = bid % nchunk;
    bid /= nchunk;
    const int64_t mt = bid % n_mtiles;
    const int64_t bh = bid / n_mtiles;
    const int64_t m = mt * blockDim.x + threadIdx.x;
    const bool active = m < M;
    const int64_t mm = active ? m : 0;

    float ar[D], gr[D], accA[MODE == 3 ? D : 1], accB[D];
    {
        const AT* ap = a + ((a_per_head ? bh % H : bh) * M + mm) * D;
        const float* gp = g + (bh * M + mm) * D;
#pragma unroll
        for (int d = 0; d < D; ++d) {
            ar[d] = operand<T>(ld_f32(ap + d)) * sl2;
            gr[d] = MODE == 3 ? operand<T>(gp[d]) : gp[d];
            accB[d] = 0.f;
            if (MODE == 3) accA[d] = 0.f;
        }
    }
    const float Lr = MODE == 3 ? 0.f : Lrow[bh * M + mm];
    const float cr = MODE == 3 ? 0.f : crow[bh * M + mm];

    const int64_t n_begin = c * chunk_len;
    const int64_t n_end = min(N, n_begin + chunk_len);
    const T* kp = kb + bh * N * D;
    const T* wp = wb + bh * N * D;
    for (int64_t n0 = n_begin; n0 < n_end; n0 += kTok) {
        const int cnt = (int)min((int64_t)kTok, n_end - n0);
        __syncthreads();
        for (int i = threadIdx.x; i < kTok * D; i += blockDim.x) {
            const int j = i / D, d = i % D;
            const bool in = j < cnt;
            ks[j][d] = in ? ld_f32(kp + (n0 + j) * D + d) : 0.f;
            ws[j][d] = in ? ld_f32(wp + (n0 + j) * D + d) : 0.f;
        }
        if (MODE == 3 && threadIdx.x < kTok) {
            const int j = threadIdx.x;
            lc[j] = j < cnt ? Lcol[bh * N + n0 + j] : 0.f;
            cc[j] = j < cnt ? ccol[bh * N + n0 + j] : 0.f;
        }
        __syncthreads();
        for (int j = 0; j < cnt; ++j) {
            float x = 0.f, dp = 0.f;
#pragma unroll
            for (int d = 0; d < D; ++d) {
                x = fmaf(ar[d], ks[j][d], x);
                dp = fmaf(gr[d], ws[j][d], dp);
            }
            const float p = ex2(x - (MODE == 3 ? lc[j] : Lr));
            const float ds = p * (dp - (MODE == 3 ? cc[j] : cr));
#pragma unroll
            for (int d = 0; d < D; ++d) {
                accB[d] = fmaf(ds, ks[j][d], accB[d]);
                if (MODE == 3) accA[d] = fmaf(p, ws[j][d], accA[d]);
            }
        }
    }
    if (active) {
        const int64_t row = (bh * nchunk + c) * M + m;
#pragma unroll
        for (int d = 0; d < D; ++d) {
            pb[row * D + d] = accB[d];
            if (MODE == 3) pa[row * D + d] = accA[d];
        }
    }
}

// Reduce of the route passes' partials, one warp per latent row, chunks in ascending order.
//   MODE 3: dZ = sum pa, dQ = s sum pb, c2 = <dZ, Z>
//   MODE 2: dQ += s sum pb, c1 = <dQ, Q>
//   MODE 1: dseeds[h, m] = s sum_b sum_chunks pb (rows = H * M)
// `op`, when not null, receives a bf16 copy of dZ (MODE 3) or dQ (MODE 2). In MODE 2 c1 is
// then taken from that copy: the passes of call 1 form dP = dQ K~^T from the bf16 dQ, and
// dS = P (dP - c1) cancels for a nearly one-hot P only when c1 = <dQ, Q> uses the same dQ.
template <int D, typename T, int MODE>
__global__ void bwd_reduce_kernel(const float* __restrict__ pa, const float* __restrict__ pb,
                                  int64_t rows, int64_t B, int64_t H, int64_t M, int64_t nchunk,
                                  float scale, const float* __restrict__ O,
                                  float* __restrict__ dz, float* __restrict__ dq,
                                  float* __restrict__ cout, T* __restrict__ dseeds,
                                  __nv_bfloat16* __restrict__ op) {
    constexpr int PER = (D + 31) / 32;
    const int lane = threadIdx.x & 31;
    const int64_t row = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
    if (row >= rows) return;
    float sa[PER], sb[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) sa[i] = sb[i] = 0.f;
    if (MODE == 1) {
        const int64_t h = row / M, m = row % M;
        for (int64_t b = 0; b < B; ++b)
            for (int64_t c = 0; c < nchunk; ++c) {
                const int64_t r = ((b * H + h) * nchunk + c) * M + m;
#pragma unroll
                for (int i = 0; i < PER; ++i) {
                    const int d = lane + 32 * i;
                    if (d < D) sb[i] += pb[r * D + d];
                }
            }
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const int d = lane + 32 * i;
            if (d < D) st_out(dseeds + row * D + d, scale * sb[i]);
        }
        return;
    }
    const int64_t bh = row / M, m = row % M;
    for (int64_t c = 0; c < nchunk; ++c) {
        const int64_t r = (bh * nchunk + c) * M + m;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const int d = lane + 32 * i;
            if (d < D) {
                sb[i] += pb[r * D + d];
                if (MODE == 3) sa[i] += pa[r * D + d];
            }
        }
    }
    float dot = 0.f;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const int d = lane + 32 * i;
        if (d < D) {
            if (MODE == 3) {
                dz[row * D + d] = sa[i];
                dq[row * D + d] = scale * sb[i];
                dot = fmaf(sa[i], O[row * D + d], dot);
                if (op) op[row * D + d] = __float2bfloat16_rn(sa[i]);
            } else {
                const float v = dq[row * D + d] + scale * sb[i];
                dq[row * D + d] = v;
                float vc = v;
                if (op) {
                    const __nv_bfloat16 vb = __float2bfloat16_rn(v);
                    op[row * D + d] = vb;
                    vc = __bfloat162float(vb);
                }
                dot = fmaf(vc, O[row * D + d], dot);
            }
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
    if (lane == 0) cout[row] = dot;
}

// Token pass; thread = token n, every route streamed.
//   MODE 23 (calls 3 and 2 together): keys k = K_n, w = V_n, y = dY_n; routes a = Q, g = dZ,
//     z = Z with L2, c2 per route and L3, c3 of the token:
//     x = s' <k, q_m>; P2 = 2^(x - L2_m); P3 = 2^(x - L3_n);
//     dS = P2 (<w, dz_m> - c2_m) + P3 (<y, z_m> - c3_n)
//     dK = s sum_m dS q_m;  dV = sum_m P2 dz_m
//   MODE 1: k = Kt_n, w = Vt_n; routes a = seeds (per head), g = dQ with L1, c1:
//     P1 = 2^(x - L1_m); dS = P1 (<w, dq_m> - c1_m); dKt = s sum_m dS a_m; dVt = sum_m P1 dq_m
// grid.x = ceil(N / 128) * BH; block = 128 threads.
template <int D, typename T, typename AT, int MODE>
__global__ void __launch_bounds__(128) token_pass_kernel(
    const T* __restrict__ kb, const T* __restrict__ wb, const T* __restrict__ yb,
    const AT* __restrict__ a, int a_per_head, const float* __restrict__ g,
    const float* __restrict__ z, const float* __restrict__ Lrow, const float* __restrict__ crow,
    const float* __restrict__ Lcol, const float* __restrict__ ccol, int64_t H, int64_t N,
    int64_t M, float sl2, float scale, T* __restrict__ dk_out, T* __restrict__ dv_out) {
    __shared__ float as_[kRoute][D];
    __shared__ float gs[kRoute][D];
    __shared__ float zs[MODE == 23 ? kRoute : 1][D];
    __shared__ float ls[kRoute], cs[kRoute];
    const int64_t ntiles = (N + 127) / 128;
    const int64_t bh = blockIdx.x / ntiles;
    const int64_t n = (blockIdx.x % ntiles) * 128 + threadIdx.x;
    const bool active = n < N;
    const int64_t nn = active ? n : 0;
    float kr[D], wr[D], yr[MODE == 23 ? D : 1], dk[D], dv[D];
#pragma unroll
    for (int d = 0; d < D; ++d) {
        kr[d] = ld_f32(kb + (bh * N + nn) * D + d) * sl2;
        wr[d] = ld_f32(wb + (bh * N + nn) * D + d);
        if (MODE == 23) yr[d] = ld_f32(yb + (bh * N + nn) * D + d);
        dk[d] = dv[d] = 0.f;
    }
    const float L3 = MODE == 23 ? Lcol[bh * N + nn] : 0.f;
    const float c3 = MODE == 23 ? ccol[bh * N + nn] : 0.f;
    const AT* ab = a + (a_per_head ? bh % H : bh) * M * D;
    const float* gb = g + bh * M * D;
    const float* zb = MODE == 23 ? z + bh * M * D : nullptr;
    for (int64_t m0 = 0; m0 < M; m0 += kRoute) {
        const int cnt = (int)min((int64_t)kRoute, M - m0);
        __syncthreads();
        for (int i = threadIdx.x; i < kRoute * D; i += blockDim.x) {
            const int j = i / D, d = i % D;
            const bool in = j < cnt;
            as_[j][d] = in ? operand<T>(ld_f32(ab + (m0 + j) * D + d)) : 0.f;
            gs[j][d] = in ? gb[(m0 + j) * D + d] : 0.f;
            if (MODE == 23) zs[j][d] = in ? operand<T>(zb[(m0 + j) * D + d]) : 0.f;
        }
        if (threadIdx.x < kRoute) {
            const int j = threadIdx.x;
            ls[j] = j < cnt ? Lrow[bh * M + m0 + j] : 0.f;
            cs[j] = j < cnt ? crow[bh * M + m0 + j] : 0.f;
        }
        __syncthreads();
        for (int j = 0; j < cnt; ++j) {
            float x = 0.f, dp = 0.f, dp3 = 0.f;
#pragma unroll
            for (int d = 0; d < D; ++d) {
                x = fmaf(kr[d], as_[j][d], x);
                dp = fmaf(wr[d], gs[j][d], dp);
                if (MODE == 23) dp3 = fmaf(yr[d], zs[j][d], dp3);
            }
            const float p = ex2(x - ls[j]);
            float ds = p * (dp - cs[j]);
            if (MODE == 23) ds = fmaf(ex2(x - L3), dp3 - c3, ds);
#pragma unroll
            for (int d = 0; d < D; ++d) {
                dk[d] = fmaf(ds, as_[j][d], dk[d]);
                dv[d] = fmaf(p, gs[j][d], dv[d]);
            }
        }
    }
    if (active) {
#pragma unroll
        for (int d = 0; d < D; ++d) {
            st_out(dk_out + (bh * N + n) * D + d, scale * dk[d]);
            st_out(dv_out + (bh * N + n) * D + d, dv[d]);
        }
    }
}

template <int D, typename T>
cudaError_t route_bwd_d(const Plan& p, const BwdPlan& bp, const T* seeds, const T* Kt,
                        const T* Vt, const T* K, const T* V, float scale, const T* Y,
                        const T* dY, const char* saved, T* dseeds, T* dKt, T* dVt, T* dK,
                        T* dV, char* ws, cudaStream_t st) {
    const SavedLayout sl = saved_layout(p);
    const float* Q32 = (const float*)(saved + sl.off_q);
    const float* Z32 = (const float*)(saved + sl.off_z);
    const float* L1 = (const float*)(saved + sl.off_l1);
    const float* L2 = (const float*)(saved + sl.off_l2);
    const float* L3 = (const float*)(saved + sl.off_l3);
    float* pa = (float*)(ws + bp.off_pa);
    float* pb = (float*)(ws + bp.off_pb);
    float* dz = (float*)(ws + bp.off_dz);
    float* dq = (float*)(ws + bp.off_dq);
    float* c1 = (float*)(ws + bp.off_d1);
    float* c2 = (float*)(ws + bp.off_d2);
    float* c3 = (float*)(ws + bp.off_d3);
    const float sl2 = scale * kLog2e;
    const int64_t tok_rows = p.BH * p.N;
    const int64_t lat_rows = p.BH * p.M;
    const unsigned route_blocks = (unsigned)(bp.nchunk * bp.n_mtiles * p.BH);
    const int route_threads = (int)bp.m_tile;
    const unsigned token_blocks = (unsigned)(((p.N + 127) / 128) * p.BH);
    const unsigned red_blocks = (unsigned)((lat_rows + 7) / 8);

    launch_delta_tokens<D, T>(dY, Y, tok_rows, c3, st);
    // call 3: dZ and the decoder's dQ
    route_pass_kernel<D, T, float, 3><<<route_blocks, route_threads, 0, st>>>(
        Q32, 0, K, dY, Z32, nullptr, nullptr, L3, c3, p.H, p.N, p.M, bp.chunk_len, bp.nchunk,
        bp.n_mtiles, sl2, pa, pb);
    bwd_reduce_kernel<D, T, 3><<<red_blocks, 256, 0, st>>>(pa, pb, lat_rows, p.B, p.H, p.M,
                                                           bp.nchunk, scale, Z32, dz, dq, c2,
                                                           nullptr, nullptr);
    // calls 3 and 2: dK and dV per token
    token_pass_kernel<D, T, float, 23><<<token_blocks, 128, 0, st>>>(
        K, V, dY, Q32, 0, dz, Z32, L2, c2, L3, c3, p.H, p.N, p.M, sl2, scale, dK, dV);
    // call 2: the encoder's dQ, added to the decoder's
    route_pass_kernel<D, T, float, 2><<<route_blocks, route_threads, 0, st>>>(
        Q32, 0, K, V, dz, L2, c2, nullptr, nullptr, p.H, p.N, p.M, bp.chunk_len, bp.nchunk,
        bp.n_mtiles, sl2, nullptr, pb);
    bwd_reduce_kernel<D, T, 2><<<red_blocks, 256, 0, st>>>(nullptr, pb, lat_rows, p.B, p.H, p.M,
                                                           bp.nchunk, scale, Q32, nullptr, dq, c1,
                                                           nullptr, nullptr);
    // call 1: dKt, dVt per token, then the seeds' gradient
    token_pass_kernel<D, T, T, 1><<<token_blocks, 128, 0, st>>>(
        Kt, Vt, nullptr, seeds, 1, dq, nullptr, L1, c1, nullptr, nullptr, p.H, p.N, p.M, sl2,
        scale, dKt, dVt);
    route_pass_kernel<D, T, T, 1><<<route_blocks, route_threads, 0, st>>>(
        seeds, 1, Kt, Vt, dq, L1, c1, nullptr, nullptr, p.H, p.N, p.M, bp.chunk_len, bp.nchunk,
        bp.n_mtiles, sl2, nullptr, pb);
    const int64_t seed_rows = p.H * p.M;
    bwd_reduce_kernel<D, T, 1><<<(unsigned)((seed_rows + 7) / 8), 256, 0, st>>>(
        nullptr, pb, seed_rows, p.B, p.H, p.M, bp.nchunk, scale, nullptr, nullptr, nullptr,
        nullptr, dseeds, nullptr);
    return cudaGetLastError();
}

// ---------------------------------------------------------------- the merged T23 pass
// T23C (tc_bwd.cu) multiplies V and dZ scaled by u = 2^(L3[n] - R) and w = 2^(R - L2[m])
// for one shift R per (b, h). With R = min_m L2 both scales stay within 2^kMergeRange
// whenever max_n L3 - R and max_m L2 - R do; a (b, h) outside that range (scores spread
// over more than ~60 binary orders) is flagged and runs the unmerged T23 pass instead.
constexpr float kMergeRange = 60.f;

// part[bh][j] for j < kRangeParts: max of L3 over slice j of the tokens; part[bh][kRangeParts]
// and [kRangeParts + 1]: min and max of L2 (from slice 0's block). One block per (bh, j).
__global__ void __launch_bounds__(256) merge_range_kernel(const float* __restrict__ L2,
                                                          const float* __restrict__ L3, int64_t M,
                                                          int64_t N, float* __restrict__ part) {
    __shared__ float red[3][8];
    const int64_t bh = blockIdx.x / kRangeParts;
    const int j = (int)(blockIdx.x % kRangeParts);
    const int64_t per = (N + kRangeParts - 1) / kRangeParts;
    const int64_t n0 = j * per, n1 = min(N, n0 + per);
    float mx3 = -INFINITY, mn2 = INFINITY, mx2 = -INFINITY;
    for (int64_t n = n0 + threadIdx.x; n < n1; n += blockDim.x) mx3 = fmaxf(mx3, L3[bh * N + n]);
    if (j == 0)
        for (int64_t m = threadIdx.x; m < M; m += blockDim.x) {
            const float x = L2[bh * M + m];
            mn2 = fminf(mn2, x);
            mx2 = fmaxf(mx2, x);
        }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        mx3 = fmaxf(mx3, __shfl_xor_sync(0xffffffffu, mx3, off));
        mn2 = fminf(mn2, __shfl_xor_sync(0xffffffffu, mn2, off));
        mx2 = fmaxf(mx2, __shfl_xor_sync(0xffffffffu, mx2, off));
    }
    const int w = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) {
        red[0][w] = mx3;
        red[1][w] = mn2;
        red[2][w] = mx2;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int k = 1; k < (int)(blockDim.x >> 5); ++k) {
            mx3 = fmaxf(mx3, red[0][k]);
            mn2 = fminf(mn2, red[1][k]);
            mx2 = fmaxf(mx2, red[2][k]);
        }
        float* o = part + bh * (kRangeParts + 2);
        o[j] = mx3;
        if (j == 0) {
            o[kRangeParts] = mn2;
            o[kRangeParts + 1] = mx2;
        }
    }
}

// R[bh] = min_m L2 and flags[bh] = 1 when the (b, h) runs the unmerged pass.
__global__ void merge_flags_kernel(const float* __restrict__ part, int64_t BH,
                                   float* __restrict__ Rb, int* __restrict__ flags) {
    const int64_t bh = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (bh >= BH) return;
    const float* o = part + bh * (kRangeParts + 2);
    float mx3 = -INFINITY;
    for (int j = 0; j < kRangeParts; ++j) mx3 = fmaxf(mx3, o[j]);
    const float R = o[kRangeParts], mx2 = o[kRangeParts + 1];
    Rb[bh] = R;
    flags[bh] = (mx3 - R <= kMergeRange && mx2 - R <= kMergeRange) ? 0 : 1;
}

// The merged pass's route operand w dZ: W[bh][m][:] = bf16(2^(R[bh] - L2[bh][m]) dZ[bh][m][:]).
__global__ void merge_operand_kernel(const float* __restrict__ dz, const float* __restrict__ L2,
                                     const float* __restrict__ Rb, int64_t M, int64_t D,
                                     int64_t total, __nv_bfloat16* __restrict__ W) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t row = i / D;  // bh * M + m
        W[i] = __float2bfloat16_rn(exp2f(Rb[row / M] - L2[row]) * dz[i]);
    }
}

// The tensor-core path (bf16 inputs): c3, the bf16 operand copies of Q and Z, then
// R3 -> reduce (dZ, the decoder's dQ, c2) -> T23 (dK, dV) and R2 -> reduce (dQ, c1) ->
// T1 (dKt, dVt) and R1 -> reduce (dseeds). For D <= 32, T23 runs merged (T23C) for every
// (b, h) whose statistics allow it and unmerged for the rest.
template <int D>
cudaError_t route_bwd_tc_d(const Plan& p, const BwdPlan& bp, const void* seeds, const void* Kt,
                           const void* Vt, const void* K, const void* V, float scale,
                           const void* Y, const void* dY, const char* saved, void* dseeds,
                           void* dKt, void* dVt, void* dK, void* dV, char* ws, cudaStream_t st) {
    using T = __nv_bfloat16;
    const SavedLayout sl = saved_layout(p);
    const float* Q32 = (const float*)(saved + sl.off_q);
    const float* Z32 = (const float*)(saved + sl.off_z);
    const float* L1 = (const float*)(saved + sl.off_l1);
    const float* L2 = (const float*)(saved + sl.off_l2);
    const float* L3 = (const float*)(saved + sl.off_l3);
    float* pa = (float*)(ws + bp.off_pa);
    float* pb = (float*)(ws + bp.off_pb);
    float* dz = (float*)(ws + bp.off_dz);
    float* dq = (float*)(ws + bp.off_dq);
    float* c1 = (float*)(ws + bp.off_d1);
    float* c2 = (float*)(ws + bp.off_d2);
    float* c3 = (float*)(ws + bp.off_d3);
    T* qb = (T*)(ws + bp.off_qb);
    T* zb = (T*)(ws + bp.off_zb);
    T* dzb = (T*)(ws + bp.off_dzb);
    T* dqb = (T*)(ws + bp.off_dqb);
    T* wop = (T*)(ws + bp.off_w);
    float* Rb = (float*)(ws + bp.off_rb);
    int* flags = (int*)(ws + bp.off_flags);
    float* rpart = (float*)(ws + bp.off_rpart);
    int* status = (int*)(ws + bp.off_status);
    const int64_t tok_rows = p.BH * p.N;
    const int64_t lat_rows = p.BH * p.M;
    const int64_t lat = lat_rows * p.D;
    const unsigned red_blocks = (unsigned)((lat_rows + 7) / 8);
    const unsigned cvt_blocks = (unsigned)min((int64_t)1024, (lat + 255) / 256);
    cudaError_t e;

    constexpr bool kMerged = D <= 32;
    launch_delta_tokens<D, T>((const T*)dY, (const T*)Y, tok_rows, c3, st);
    // Q as the training forward gave it to calls 2 and 3: a hi/lo pair for D <= 32
    T* qlo = kMerged ? (T*)(ws + bp.off_qlo) : nullptr;
    if (qlo)
        to_bf16_hilo_kernel<<<cvt_blocks, 256, 0, st>>>(Q32, qb, qlo, lat);
    else
        to_bf16_kernel<<<cvt_blocks, 256, 0, st>>>(Q32, qb, lat);
    to_bf16_kernel<<<cvt_blocks, 256, 0, st>>>(Z32, zb, lat);
    if (kMerged) {
        merge_range_kernel<<<(unsigned)(p.BH * kRangeParts), 256, 0, st>>>(L2, L3, p.M, p.N,
                                                                           rpart);
        merge_flags_kernel<<<(unsigned)((p.BH + 127) / 128), 128, 0, st>>>(rpart, p.BH, Rb,
                                                                            flags);
    }
    TcBwdOperands o{};
    // R3: route rows; S = Q K^T, dP = Z dY^T; column statistics L3, c3 -> dQ3, dZ partials
    o = TcBwdOperands{{qb, zb, zb}, {K, dY, dY}, nullptr, nullptr, L3, c3, pa, pb, nullptr,
                      nullptr};
    o.lo = qlo;
    if ((e = tc_bwd_pass(p, bp, 0, o, scale, status, st)) != cudaSuccess) return e;
    bwd_reduce_kernel<D, T, 3><<<red_blocks, 256, 0, st>>>(pa, pb, lat_rows, p.B, p.H, p.M,
                                                           bp.nchunk, scale, Z32, dz, dq, c2,
                                                           nullptr, dzb);
    // T23: token rows; S = K Q^T, dP2 = V dZ^T, dP3 = dY Z^T -> dK, dV
    o = TcBwdOperands{{K, V, dY}, {qb, dzb, zb}, L3, c3, L2, c2, nullptr, nullptr, dK, dV};
    o.lo = qlo;
    if (kMerged) {
        // T23C: S = K Q^T, T = dY Z^T + (u V) (w dZ)^T; the flagged (b, h) run T23 after it
        merge_operand_kernel<<<cvt_blocks, 256, 0, st>>>(dz, L2, Rb, p.M, p.D, lat, wop);
        TcBwdOperands om{{K, dY, V}, {qb, wop, zb}, L3, c3, L2, c2, nullptr, nullptr, dK, dV};
        om.Rb = Rb;
        om.flags = flags;
        om.want = 0;
        om.lo = qlo;
        if ((e = tc_bwd_pass(p, bp, 5, om, scale, status, st)) != cudaSuccess) return e;
        o.flags = flags;
        o.want = 1;
    }
    if ((e = tc_bwd_pass(p, bp, 3, o, scale, status, st)) != cudaSuccess) return e;
    // R2: route rows; S = Q K^T, dP = dZ V^T; row statistics L2, c2 -> dQ2 partials
    o = TcBwdOperands{{qb, dzb, dzb}, {K, V, V}, L2, c2, nullptr, nullptr, nullptr, pb, nullptr,
                      nullptr};
    o.lo = qlo;
    if ((e = tc_bwd_pass(p, bp, 1, o, scale, status, st)) != cudaSuccess) return e;
    bwd_reduce_kernel<D, T, 2><<<red_blocks, 256, 0, st>>>(nullptr, pb, lat_rows, p.B, p.H, p.M,
                                                           bp.nchunk, scale, Q32, nullptr, dq, c1,
                                                           nullptr, dqb);
    // T1: token rows; S = Kt Qs^T, dP = Vt dQ^T; column statistics L1, c1 -> dKt, dVt
    o = TcBwdOperands{{Kt, Vt, Vt}, {seeds, dqb, dqb}, nullptr, nullptr, L1, c1, nullptr,
                      nullptr, dKt, dVt};
    if ((e = tc_bwd_pass(p, bp, 4, o, scale, status, st)) != cudaSuccess) return e;
    // R1: route rows; S = Qs Kt^T, dP = dQ Vt^T; row statistics L1, c1 -> dQs partials
    o = TcBwdOperands{{seeds, dqb, dqb}, {Kt, Vt, Vt}, L1, c1, nullptr, nullptr, nullptr, pb,
                      nullptr, nullptr};
    if ((e = tc_bwd_pass(p, bp, 2, o, scale, status, st)) != cudaSuccess) return e;
    const int64_t seed_rows = p.H * p.M;
    bwd_reduce_kernel<D, T, 1><<<(unsigned)((seed_rows + 7) / 8), 256, 0, st>>>(
        nullptr, pb, seed_rows, p.B, p.H, p.M, bp.nchunk, scale, nullptr, nullptr, nullptr,
        nullptr, (T*)dseeds, nullptr);
    return cudaGetLastError();
}

template <typename T>
cudaError_t route_bwd_t(const Plan& p, const BwdPlan& bp, const void* seeds, const void* Kt,
                        const void* Vt, const void* K, const void* V, float scale, const void* Y,
                        const void* dY, const char* saved, void* dseeds, void* dKt, void* dVt,
                        void* dK, void* dV, char* ws, cudaStream_t st) {
#define FLAREPP_BWD(DD)                                                                          \
    return route_bwd_d<DD, T>(p, bp, (const T*)seeds, (const T*)Kt, (const T*)Vt, (const T*)K,  \
                              (const T*)V, scale, (const T*)Y, (const T*)dY, saved, (T*)dseeds, \
                              (T*)dKt, (T*)dVt, (T*)dK, (T*)dV, ws, st);
    switch (p.D) {
        case 16: FLAREPP_BWD(16)
        case 32: FLAREPP_BWD(32)
        case 64: FLAREPP_BWD(64)
        default: return cudaErrorInvalidValue;
    }
#undef FLAREPP_BWD
}

}  // namespace

cudaError_t route_bwd(const Plan& p, const BwdPlan& bp, const void* seeds, const void* Kt,
                      const void* Vt, const void* K, const void* V, float scale, const void* Y,
                      const void* dY, const char* saved, void* dseeds, void* dKt, void* dVt,
                      void* dK, void* dV, char* ws, cudaStream_t st) {
    if (bp.path == kPathTc) {
#define FLAREPP_TCBWD(DD)                                                                     \
    return route_bwd_tc_d<DD>(p, bp, seeds, Kt, Vt, K, V, scale, Y, dY, saved, dseeds, dKt, \
                              dVt, dK, dV, ws, st);
        switch (p.D) {
            case 16: FLAREPP_TCBWD(16)
            case 32: FLAREPP_TCBWD(32)
            case 64: FLAREPP_TCBWD(64)
            default: return cudaErrorInvalidValue;
        }
#undef FLAREPP_TCBWD
    }
    return route_bwd_t<float>(p, bp, seeds, Kt, Vt, K, V, scale, Y, dY, saved, dseeds, dKt, dVt,
                              dK, dV, ws, st);
}

}  // namespace flarepp
