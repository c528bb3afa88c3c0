// Tensor-core (tcgen05 / TMEM / TMA) GEMMs of the FLARE++ mixer's pointwise projections
// (Fig. 1; eqs. flarepp_query_synthesis and flarepp_mixer): out = A B^T with bf16 operands,
// float32 accumulation in TMEM and bf16 results written by a layout-aware epilogue.
//
//   projection (MODE 0): A = X [B][N][C] (token rows), B = W_in [P*C][C] (out x in). The P*C
//     output channels of a token are the projections K, V, K~, V~ (P = 4; P = 2 for the shared
//     projection), each split into H heads of width D and written to its [B][H][N][D] tensor,
//     the layout the routing chain reads.
//   output (MODE 1): A = merge(Y), read head by head straight from Y [B][H][N][D] (no merged
//     copy is made), B = Wo [C][C]; O [B][N][C].
//
// The contraction over C runs in slices of D channels (one head), the unit that both A
// layouts share; each slice is one TMA box of 128 tokens x D for A and NT channels x D for B,
// swizzled to the D-wide row. A work tile is 128 tokens (of one batch element) x NT output
// channels; persistent CTAs walk the tiles with the channel tile varying fastest, so the CTAs
// that share a token tile run together and read it from L2.
//
// Roles (12 warps): warp 0 the TMA producer, warp 1 the MMA issuer (one elected lane; one
// commit per slice frees its ring stage, one per tile hands the accumulator over), warps 4..11
// two epilogue warpgroups (TMEM lane = token row; each takes half of the tile's channels). Two TMEM accumulators of NT <= 256 columns let the
// epilogue of one tile overlap the products of the next. Every wait is bounded (2 s of
// %globaltimer): on expiry the kernel records FLAREPP_ERR_TIMEOUT in the status word, every
// role leaves its loops, the producer waits for its copies in flight, the MMA issuer for its
// products, and TMEM is freed.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <math.h>
#include <mutex>

#include "flarepp_internal.h"
#include "tc_ptx.cuh"

namespace flarepp {
namespace {

using namespace tc;

constexpr int kEpiGroups = 2;  // epilogue warpgroups; each takes half of a tile's channels
constexpr int kThreads = (4 + 4 * kEpiGroups) * 32;
constexpr int kFirstEpiWarp = 4;
constexpr int kRows = 128;    // tokens per tile (TMEM lanes, MMA M)
constexpr int kMaxNT = 256;   // output channels per tile, at most
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint32_t kTmemCols = 512;

template <int D>
struct GCfg {
    static constexpr int kASlice = kRows * D * 2;
    static constexpr int kBSlice = kMaxNT * D * 2;
    static constexpr int kStage = kASlice + kBSlice;
    static constexpr int kStages = (192 * 1024) / kStage > 8 ? 8 : (192 * 1024) / kStage;
    static constexpr uint32_t kSwz = D == 16 ? kSw32 : (D == 32 ? kSw64 : kSw128);
    static constexpr uint32_t kSBO = 8 * D * 2;
    static constexpr int kNumBars = 2 * kStages + 4 + 1;  // full, empty, accfull[2], accempty[2], fin
    static constexpr int kNeed = 1024 + kStages * kStage + kNumBars * 8 + 16;
    static constexpr int kSmem = kNeed > 122880 ? kNeed : 122880;  // one CTA per SM
    static_assert(kSmem <= 232448, "shared memory budget");
};

struct GemmParams {
    int64_t B, N, H, C;
    int64_t n_out;      // output channels (P * C, or C)
    int NT;             // output channels per tile (a multiple of 16, <= 256, divides C)
    uint32_t idesc;     // MMA instruction descriptor for M = 128, N = NT
    int64_t row_tiles;  // 128-token tiles per batch element
    int64_t col_tiles;  // n_out / NT
    int64_t n_tiles;
    __nv_bfloat16* out[4];  // MODE 0: the P [B][H][N][D] tensors; MODE 1: O [B][N][C]
    int* status;
};

struct GTile {
    int64_t b, rt, ct;
};

__device__ __forceinline__ GTile gtile(const GemmParams& p, int64_t t) {
    GTile T;
    T.ct = t % p.col_tiles;
    const int64_t r = t / p.col_tiles;
    T.rt = r % p.row_tiles;
    T.b = r / p.row_tiles;
    return T;
}

__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                         int* status) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 63u) == 0) {
            if (*abort_flag) return false;
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                *abort_flag = 1;
                atomicExch(status, (int)FLAREPP_ERR_TIMEOUT);
                return false;
            }
        }
    }
}
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          int* status) {
    const bool got = wait_bar(bar, parity, abort_flag, status);
    return __all_sync(0xffffffffu, got);
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

template <int D, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const GemmParams prm) {
    using C = GCfg<D>;
    constexpr int kS = C::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kS * C::kStage);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::kNumBars);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t full0 = smem_u32(bars);
    const uint32_t empty0 = full0 + 8u * kS;
    const uint32_t accfull0 = empty0 + 8u * kS;
    const uint32_t accempty0 = accfull0 + 16u;
    const uint32_t fin = accempty0 + 16u;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int slices = (int)(prm.C / D);

    if (threadIdx.x == 0) {
        for (int st = 0; st < kS; ++st) {
            mbar_init(full0 + 8u * st, 1);
            mbar_init(empty0 + 8u * st, 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accfull0 + 8u * b, 1);
            mbar_init(accempty0 + 8u * b, kRows * kEpiGroups);
        }
        mbar_init(fin, 1);
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmA);
        prefetch_tmap(&tmB);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        uint32_t it = 0;
        bool ok = true;
        const uint32_t bytes = (uint32_t)(C::kASlice + prm.NT * D * 2);
        for (int64_t t = blockIdx.x; t < prm.n_tiles && ok; t += gridDim.x) {
            const GTile T = gtile(prm, t);
            for (int h = 0; h < slices; ++h, ++it) {
                const int st = it % kS;
                if (it >= (uint32_t)kS &&
                    !warp_wait(empty0 + 8u * st, ((it / kS) - 1) & 1, abort_flag, prm.status)) {
                    ok = false;
                    break;
                }
                if (elect_one()) {
                    const uint32_t dst = smem_u32(smem + st * C::kStage);
                    mbar_expect_tx(full0 + 8u * st, bytes);
                    if (MODE == 0)
                        tma_load_3d(dst, &tmA, h * D, (int)(T.rt * kRows), (int)T.b,
                                    full0 + 8u * st);
                    else
                        tma_load_3d(dst, &tmA, 0, (int)(T.rt * kRows), (int)(T.b * prm.H + h),
                                    full0 + 8u * st);
                    tma_load_3d(dst + C::kASlice, &tmB, h * D, (int)(T.ct * prm.NT), 0,
                                full0 + 8u * st);
                }
                __syncwarp();
            }
        }
        if (!ok) {  // wait (bounded) until every copy issued has landed
            const uint64_t t0 = globaltimer_ns();
            for (int st = 0; st < kS && (uint32_t)st < it; ++st) {
                const uint32_t x = it - 1 - ((it - 1 - st) % kS);
                while (!mbar_try_wait(full0 + 8u * st, (x / kS) & 1) &&
                       globaltimer_ns() - t0 < kWaitLimitNs) {
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        uint32_t it = 0, j = 0;
        bool ok = true;
        for (int64_t t = blockIdx.x; t < prm.n_tiles && ok; t += gridDim.x, ++j) {
            const int ab = j & 1;
            if (j >= 2 &&
                !warp_wait(accempty0 + 8u * ab, ((j >> 1) - 1) & 1, abort_flag, prm.status)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t acc = tmem + ab * kMaxNT;
            for (int h = 0; h < slices; ++h, ++it) {
                const int st = it % kS;
                if (!warp_wait(full0 + 8u * st, (it / kS) & 1, abort_flag, prm.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a = smem_u32(smem + st * C::kStage);
                const uint32_t b = a + C::kASlice;
#pragma unroll
                for (int k = 0; k < D / 16; ++k) {
                    const uint64_t ad = smem_desc(a + 32 * k, 16, C::kSBO, C::kSwz);
                    const uint64_t bd = smem_desc(b + 32 * k, 16, C::kSBO, C::kSwz);
                    if (elect_one()) mma_ss(acc, ad, bd, prm.idesc, (h > 0 || k > 0) ? 1u : 0u);
                    __syncwarp();
                }
                if (elect_one()) mma_commit(empty0 + 8u * st);  // the slice's stage is free
                __syncwarp();
            }
            if (!ok) break;
            if (elect_one()) mma_commit(accfull0 + 8u * ab);
            __syncwarp();
        }
        if (elect_one()) mma_commit(fin);
        __syncwarp();
        const uint64_t tw = globaltimer_ns();
        while (!__all_sync(0xffffffffu, mbar_try_wait(fin, 0)) &&
               globaltimer_ns() - tw < kWaitLimitNs) {
        }
    } else if (warp >= kFirstEpiWarp) {
        // ------------------------------------------------------------ epilogue
        // Warpgroup e takes channels [e * NT / 2, (e + 1) * NT / 2) of each tile, 64 columns
        // per TMEM round (four loads, one wait).
        const int q = warp % 4;
        const int e = (warp - kFirstEpiWarp) / 4;
        const int r = 32 * q + lane;
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        const int half = prm.NT / kEpiGroups;
        uint32_t j = 0;
        for (int64_t t = blockIdx.x; t < prm.n_tiles; t += gridDim.x, ++j) {
            const GTile T = gtile(prm, t);
            const int ab = j & 1;
            if (!warp_wait(accfull0 + 8u * ab, (j >> 1) & 1, abort_flag, prm.status)) break;
            tc_fence_after();
            const int64_t n = T.rt * kRows + r;
            const bool valid = n < prm.N;
            const uint32_t acc = tmem + lane_off + ab * kMaxNT;
            // the tile's channels lie in one projection (NT divides C): its base pointer once
            const int64_t c0 = T.ct * prm.NT + e * half;
            const int64_t p = c0 / prm.C, cc0 = c0 % prm.C;
            __nv_bfloat16* base = MODE != 0 ? prm.out[0]
                                  : p == 0   ? prm.out[0]
                                  : p == 1   ? prm.out[1]
                                  : p == 2   ? prm.out[2]
                                             : prm.out[3];
            __nv_bfloat16* row = MODE == 0 ? base + (T.b * prm.H * prm.N + n) * D
                                           : base + (T.b * prm.N + n) * prm.C + c0;
            for (int c64 = 0; c64 < half; c64 += 64) {
                const int w = half - c64 < 64 ? half - c64 : 64;  // 16, 32 or 64 columns
                uint32_t v[64];
                const uint32_t col = acc + e * half + c64;
                tmem_ld16(col, v);
                if (w > 16) tmem_ld16(col + 16, v + 16);
                if (w > 32) {
                    tmem_ld16(col + 32, v + 32);
                    tmem_ld16(col + 48, v + 48);
                }
                // waits that name the loaded registers, so that no use moves above them
                tmem_wait_ld16(v);
                if (w > 16) tmem_wait_ld16(v + 16);
                if (w > 32) {
                    tmem_wait_ld16(v + 32);
                    tmem_wait_ld16(v + 48);
                }
                if (!valid) continue;
#pragma unroll
                for (int g = 0; g < 8; ++g) {
                    if (8 * g >= w) break;
                    uint4 o;
                    o.x = pack_bf16(__uint_as_float(v[8 * g + 0]), __uint_as_float(v[8 * g + 1]));
                    o.y = pack_bf16(__uint_as_float(v[8 * g + 2]), __uint_as_float(v[8 * g + 3]));
                    o.z = pack_bf16(__uint_as_float(v[8 * g + 4]), __uint_as_float(v[8 * g + 5]));
                    o.w = pack_bf16(__uint_as_float(v[8 * g + 6]), __uint_as_float(v[8 * g + 7]));
                    __nv_bfloat16* dst;
                    if (MODE == 0) {
                        const int64_t cc = cc0 + c64 + 8 * g;  // channel within the projection
                        dst = row + (cc / D) * prm.N * D + (cc % D);
                    } else {
                        dst = row + c64 + 8 * g;
                    }
                    *reinterpret_cast<uint4*>(dst) = o;
                }
            }
            tc_fence_before();
            mbar_arrive(accempty0 + 8u * ab);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// ------------------------------------------------------------------ host side

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// A bf16 tensor of dims {inner, rows, z} (inner contiguous), boxes of D x box_rows x 1,
// swizzled to the D-wide row.
bool make_map(CUtensorMap* m, const void* base, int64_t D, int64_t inner, int64_t rows,
              int64_t z, uint32_t box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)inner, (cuuint64_t)rows, (cuuint64_t)z};
    cuuint64_t strides[2] = {(cuuint64_t)(inner * 2), (cuuint64_t)(rows * inner * 2)};
    cuuint32_t box[3] = {(cuuint32_t)D, box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    const CUtensorMapSwizzle sw = D == 16 ? CU_TENSOR_MAP_SWIZZLE_32B
                                          : (D == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                     : CU_TENSOR_MAP_SWIZZLE_128B);
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D, int MODE>
cudaError_t launch(const CUtensorMap& a, const CUtensorMap& b, const GemmParams& prm,
                   cudaStream_t st) {
    using Cf = GCfg<D>;
    static cudaError_t attr = cudaFuncSetAttribute(
        tc_gemm_kernel<D, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cf::kSmem);
    if (attr != cudaSuccess) return attr;
    if (prm.n_tiles == 0) return cudaSuccess;
    int dev = 0, sms = kNumSMs;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t grid = prm.n_tiles < sms ? prm.n_tiles : sms;
    tc_gemm_kernel<D, MODE><<<(unsigned)grid, kThreads, Cf::kSmem, st>>>(a, b, prm);
    return cudaGetLastError();
}

// output channels per tile: the largest of 256, 128, 64, 32, 16 that divides C
int tile_channels(int64_t C) {
    for (int nt = kMaxNT; nt >= 16; nt /= 2)
        if (C % nt == 0) return nt;
    return 0;
}

}  // namespace

cudaError_t tc_projection(int64_t B, int64_t N, int64_t H, int64_t D, int P, const void* X,
                          const void* W_in, void* const* outs, int* status, cudaStream_t st) {
    const int64_t C = H * D;
    GemmParams prm{};
    prm.B = B;
    prm.N = N;
    prm.H = H;
    prm.C = C;
    prm.n_out = P * C;
    prm.NT = tile_channels(C);
    if (prm.NT == 0) return cudaErrorInvalidValue;
    prm.idesc = idesc_bf16_f32(kRows, prm.NT, false, false);
    prm.row_tiles = (N + kRows - 1) / kRows;
    prm.col_tiles = prm.n_out / prm.NT;
    prm.n_tiles = B * prm.row_tiles * prm.col_tiles;
    for (int p = 0; p < 4; ++p) prm.out[p] = (__nv_bfloat16*)outs[p < P ? p : 0];
    prm.status = status;
    CUtensorMap ma, mb;
    if (!make_map(&ma, X, D, C, N, B, kRows) ||
        !make_map(&mb, W_in, D, C, prm.n_out, 1, (uint32_t)prm.NT))
        return cudaErrorInvalidValue;
    switch (D) {
        case 16: return launch<16, 0>(ma, mb, prm, st);
        case 32: return launch<32, 0>(ma, mb, prm, st);
        case 64: return launch<64, 0>(ma, mb, prm, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t tc_output_projection(int64_t B, int64_t N, int64_t H, int64_t D, const void* Y,
                                 const void* Wo, void* O, int* status, cudaStream_t st) {
    const int64_t C = H * D;
    GemmParams prm{};
    prm.B = B;
    prm.N = N;
    prm.H = H;
    prm.C = C;
    prm.n_out = C;
    prm.NT = tile_channels(C);
    if (prm.NT == 0) return cudaErrorInvalidValue;
    prm.idesc = idesc_bf16_f32(kRows, prm.NT, false, false);
    prm.row_tiles = (N + kRows - 1) / kRows;
    prm.col_tiles = C / prm.NT;
    prm.n_tiles = B * prm.row_tiles * prm.col_tiles;
    prm.out[0] = prm.out[1] = prm.out[2] = prm.out[3] = (__nv_bfloat16*)O;
    prm.status = status;
    CUtensorMap ma, mb;
    if (!make_map(&ma, Y, D, D, N, B * H, kRows) ||
        !make_map(&mb, Wo, D, C, C, 1, (uint32_t)prm.NT))
        return cudaErrorInvalidValue;
    switch (D) {
        case 16: return launch<16, 1>(ma, mb, prm, st);
        case 32: return launch<32, 1>(ma, mb, prm, st);
        case 64: return launch<64, 1>(ma, mb, prm, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace flarepp
