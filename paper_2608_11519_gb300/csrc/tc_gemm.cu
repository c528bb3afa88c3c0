// Tensor-core (tcgen05 / TMEM / TMA) GEMMs of the FLARE++ mixer's pointwise projections
// (Fig. 1; eqs. flarepp_query_synthesis and flarepp_mixer): out = A B^T with bf16 operands,
// float32 accumulation in TMEM and bf16 results written by a layout-aware epilogue.
//
//   projection (MODE 0): A = X [B][N][C] (token rows), B = W_in [P*C][C] (out x in). The P*C
//     output channels of a token are the projections K, V, K~, V~ (P = 4; P = 2 for the shared
//     projection), each split into H heads of width D and written to its [B][H][N][D] tensor,
//     the layout the routing chain reads.
//   output (MODE 1): A = merge(Y), read head by head straight from Y [B][H][N][D] (no merged
//     copy is made), B = Wo [C][C]; O [B][N][C]. The same pass with up to four A tensors side
//     by side (A channel p*C + h*D + d from tensor p) computes dX = sum_p dP_p W_p of the
//     mixer's backward with B = W_in^T.
//
// The contraction over C runs in slices of D channels (one head), the unit that both A
// layouts share; each slice is one TMA box of 128 tokens x D for A and NT channels x D for B,
// swizzled to the D-wide row. A work tile is 128 tokens (of one batch element) x NT output
// channels; persistent CTAs walk the tiles with the channel tile varying fastest, so the CTAs
// that share a token tile run together and read it from L2.
//
// Roles (12 warps): warp 0 the TMA producer, warp 1 the MMA issuer (one elected lane; one
// commit per slice frees its ring stage, one per tile hands the accumulator over), warps 4..11
// two epilogue warpgroups (TMEM lane = token row; each takes every other head of the tile and
// writes it with one TMA store per head from a shared-memory staging block). Two TMEM accumulators of NT <= 256 columns let the
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
    static constexpr int kStages = (160 * 1024) / kStage > 8 ? 8 : (160 * 1024) / kStage;
    static constexpr uint32_t kSwz = D == 16 ? kSw32 : (D == 32 ? kSw64 : kSw128);
    static constexpr uint32_t kSBO = 8 * D * 2;
    // per epilogue warpgroup: its heads of one tile, [head][128 rows][D] bf16, for TMA stores
    static constexpr int kStaging = (kMaxNT / 2) * kRows * 2;
    // full, empty, accfull[2], accempty[2], fin, then per epilogue warpgroup staging_free and
    // staging_written
    static constexpr int kNumBars = 2 * kStages + 4 + 1 + 2 * kEpiGroups;
    static constexpr int kNeed =
        1024 + kStages * kStage + kEpiGroups * kStaging + kNumBars * 8 + 16;
    static constexpr int kSmem = kNeed > 122880 ? kNeed : 122880;  // one CTA per SM
    static_assert(kSmem <= 232448, "shared memory budget");
};

struct GemmParams {
    int64_t B, N, H, C;
    int n_a;            // MODE 1: A tensors side by side (the contraction runs over n_a * C)
    int64_t n_out;      // output channels (P * C, or C)
    int NT;             // output channels per tile (whole heads, <= 256, divides C)
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
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmA1,
                   const __grid_constant__ CUtensorMap tmA2, const __grid_constant__ CUtensorMap tmA3,
                   const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmO0, const __grid_constant__ CUtensorMap tmO1,
                   const __grid_constant__ CUtensorMap tmO2, const __grid_constant__ CUtensorMap tmO3,
                   const GemmParams prm) {
    using C = GCfg<D>;
    constexpr int kS = C::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    uint8_t* staging = smem + kS * C::kStage;  // [kEpiGroups][kStaging]
    uint64_t* bars = reinterpret_cast<uint64_t*>(staging + kEpiGroups * C::kStaging);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::kNumBars);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t full0 = smem_u32(bars);
    const uint32_t empty0 = full0 + 8u * kS;
    const uint32_t accfull0 = empty0 + 8u * kS;
    const uint32_t accempty0 = accfull0 + 16u;
    const uint32_t fin = accempty0 + 16u;
    const uint32_t sfree0 = fin + 8u;                      // [kEpiGroups], count 1
    const uint32_t swritten0 = sfree0 + 8u * kEpiGroups;   // [kEpiGroups], count 128
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int slices = (int)(prm.C / D) * (MODE == 1 ? prm.n_a : 1);

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
        for (int e = 0; e < kEpiGroups; ++e) {
            mbar_init(sfree0 + 8u * e, 1);
            mbar_init(swritten0 + 8u * e, kRows);
        }
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmA);
        if (MODE == 1 && prm.n_a > 1) {
            prefetch_tmap(&tmA1);
            prefetch_tmap(&tmA2);
            prefetch_tmap(&tmA3);
        }
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
                    if (MODE == 0) {
                        tma_load_3d(dst, &tmA, h * D, (int)(T.rt * kRows), (int)T.b,
                                    full0 + 8u * st);
                    } else {
                        // slice h: head h % H of A tensor h / H
                        const int p = h / (int)prm.H, hh = h % (int)prm.H;
                        const CUtensorMap* ma = p == 0 ? &tmA : p == 1 ? &tmA1 : p == 2 ? &tmA2 : &tmA3;
                        tma_load_3d(dst, ma, 0, (int)(T.rt * kRows), (int)(T.b * prm.H + hh),
                                    full0 + 8u * st);
                    }
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
        // Warpgroup e takes the tile's heads e, e + 2, ...: each head's 128 x D block goes from
        // TMEM through shared memory ([128 rows][D], one row per thread) to one TMA tensor
        // store (rows beyond N are clipped by the store). Two mbarriers per warpgroup order the
        // staging buffer (bounded waits): staging_free, which the leader arrives on once its
        // previous stores have read the buffer, and staging_written, on which every thread
        // arrives after its rows (and a proxy fence) and which the leader waits for before it
        // issues the stores.
        const int q = warp % 4;
        const int e = (warp - kFirstEpiWarp) / 4;
        const int r = 32 * q + lane;
        const bool leader = q == 0 && lane == 0;
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        const int heads = prm.NT / D;
        uint8_t* stg = staging + e * C::kStaging;
        uint32_t j = 0;
        bool pending = false;
        for (int64_t t = blockIdx.x; t < prm.n_tiles; t += gridDim.x, ++j) {
            const GTile T = gtile(prm, t);
            const int ab = j & 1;
            if (!warp_wait(accfull0 + 8u * ab, (j >> 1) & 1, abort_flag, prm.status)) break;
            tc_fence_after();
            if (pending) {
                if (leader) {
                    bulk_wait_read();
                    mbar_arrive(sfree0 + 8u * e);
                }
                if (!warp_wait(sfree0 + 8u * e, (j - 1) & 1, abort_flag, prm.status)) break;
            }
            const uint32_t acc = tmem + lane_off + ab * kMaxNT;
            int slot = 0;
            for (int hh = e; hh < heads; hh += kEpiGroups, ++slot) {
                uint32_t v[D];
#pragma unroll
                for (int k = 0; k < D / 16; ++k) tmem_ld16(acc + hh * D + 16 * k, v + 16 * k);
#pragma unroll
                for (int k = 0; k < D / 16; ++k) tmem_wait_ld16(v + 16 * k);
                // the block is stored swizzled like the operands (16-byte chunk g of row r at
                // g ^ (bits 7.. of the row's byte offset)), which the store map undoes: one
                // thread per row then writes without shared-memory bank conflicts
                uint4* dst = reinterpret_cast<uint4*>(stg + ((size_t)slot * kRows + r) * D * 2);
                const int sw = ((r * D * 2) >> 7) & (D / 8 - 1);
#pragma unroll
                for (int g = 0; g < D / 8; ++g) {
                    uint4 o;
                    o.x = pack_bf16(__uint_as_float(v[8 * g + 0]), __uint_as_float(v[8 * g + 1]));
                    o.y = pack_bf16(__uint_as_float(v[8 * g + 2]), __uint_as_float(v[8 * g + 3]));
                    o.z = pack_bf16(__uint_as_float(v[8 * g + 4]), __uint_as_float(v[8 * g + 5]));
                    o.w = pack_bf16(__uint_as_float(v[8 * g + 6]), __uint_as_float(v[8 * g + 7]));
                    dst[g ^ sw] = o;
                }
            }
            tc_fence_before();
            mbar_arrive(accempty0 + 8u * ab);  // the accumulator is read out
            fence_proxy_async();
            mbar_arrive(swritten0 + 8u * e);
            if (q == 0 && !warp_wait(swritten0 + 8u * e, j & 1, abort_flag, prm.status)) break;
            if (leader) {
                slot = 0;
                const int n0 = (int)(T.rt * kRows);
                for (int hh = e; hh < heads; hh += kEpiGroups, ++slot) {
                    const int64_t c = T.ct * prm.NT + (int64_t)hh * D;  // first channel
                    const uint32_t src = smem_u32(stg + (size_t)slot * kRows * D * 2);
                    if (MODE == 0) {
                        const int64_t p = c / prm.C, h = (c % prm.C) / D;
                        const CUtensorMap* m = p == 0 ? &tmO0 : p == 1 ? &tmO1 : p == 2 ? &tmO2 : &tmO3;
                        tma_store_3d(m, src, 0, n0, (int)(T.b * prm.H + h));
                    } else {
                        tma_store_3d(&tmO0, src, (int)c, n0, (int)T.b);
                    }
                }
                bulk_commit();
            }
            pending = true;
        }
        if (leader) bulk_wait_all();
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
cudaError_t launch(const CUtensorMap* a, const CUtensorMap& b, const CUtensorMap* o,
                   const GemmParams& prm, cudaStream_t st) {
    using Cf = GCfg<D>;
    const cudaError_t attr = ensure_smem_limit((const void*)tc_gemm_kernel<D, MODE>, Cf::kSmem);
    if (attr != cudaSuccess) return attr;
    if (prm.n_tiles == 0) return cudaSuccess;
    int dev = 0, sms = kNumSMs;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t grid = prm.n_tiles < sms ? prm.n_tiles : sms;
    tc_gemm_kernel<D, MODE><<<(unsigned)grid, kThreads, Cf::kSmem, st>>>(
        a[0], a[1], a[2], a[3], b, o[0], o[1], o[2], o[3], prm);
    return cudaGetLastError();
}

// output channels per tile: D times the largest power of two of heads that divides H and
// keeps the tile within 256 channels
int tile_channels(int64_t H, int64_t D) {
    int heads = 1;
    while (heads * 2 * D <= kMaxNT && H % (heads * 2) == 0) heads *= 2;
    return (int)(heads * D);
}

// A bf16 tensor of dims {inner, rows, z}, boxes of box_inner x 128 x 1 (the epilogue's
// staged blocks), swizzled in shared memory to the box_inner-wide row.
bool make_store_map(CUtensorMap* m, void* base, int64_t inner, int64_t rows, int64_t z,
                    uint32_t box_inner) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)inner, (cuuint64_t)rows, (cuuint64_t)z};
    cuuint64_t strides[2] = {(cuuint64_t)(inner * 2), (cuuint64_t)(rows * inner * 2)};
    cuuint32_t box[3] = {box_inner, (cuuint32_t)kRows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    const CUtensorMapSwizzle sw = box_inner == 16 ? CU_TENSOR_MAP_SWIZZLE_32B
                                  : (box_inner == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                     : CU_TENSOR_MAP_SWIZZLE_128B);
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_NONE,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
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
    prm.NT = tile_channels(H, D);
    prm.idesc = idesc_bf16_f32(kRows, prm.NT, false, false);
    prm.row_tiles = (N + kRows - 1) / kRows;
    prm.col_tiles = prm.n_out / prm.NT;
    prm.n_tiles = B * prm.row_tiles * prm.col_tiles;
    for (int p = 0; p < 4; ++p) prm.out[p] = (__nv_bfloat16*)outs[p < P ? p : p - 2];
    prm.status = status;
    CUtensorMap ma[4], mb, mo[4];
    if (!make_map(&ma[0], X, D, C, N, B, kRows) ||
        !make_map(&mb, W_in, D, C, prm.n_out, 1, (uint32_t)prm.NT))
        return cudaErrorInvalidValue;
    ma[1] = ma[2] = ma[3] = ma[0];
    prm.n_a = 1;
    for (int p = 0; p < 4; ++p)
        if (!make_store_map(&mo[p], prm.out[p], D, N, B * H, (uint32_t)D))
            return cudaErrorInvalidValue;
    switch (D) {
        case 16: return launch<16, 0>(ma, mb, mo, prm, st);
        case 32: return launch<32, 0>(ma, mb, mo, prm, st);
        case 64: return launch<64, 0>(ma, mb, mo, prm, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t tc_output_projection(int64_t B, int64_t N, int64_t H, int64_t D, const void* Y,
                                 const void* Wo, void* O, int* status, cudaStream_t st) {
    const void* ys[1] = {Y};
    return tc_heads_projection(B, N, H, D, 1, ys, Wo, O, status, st);
}

cudaError_t tc_heads_projection(int64_t B, int64_t N, int64_t H, int64_t D, int n_a,
                                const void* const* As, const void* W, void* O, int* status,
                                cudaStream_t st) {
    const int64_t C = H * D;
    if (n_a < 1 || n_a > 4) return cudaErrorInvalidValue;
    GemmParams prm{};
    prm.B = B;
    prm.N = N;
    prm.H = H;
    prm.C = C;
    prm.n_a = n_a;
    prm.n_out = C;
    prm.NT = tile_channels(H, D);
    prm.idesc = idesc_bf16_f32(kRows, prm.NT, false, false);
    prm.row_tiles = (N + kRows - 1) / kRows;
    prm.col_tiles = C / prm.NT;
    prm.n_tiles = B * prm.row_tiles * prm.col_tiles;
    prm.out[0] = prm.out[1] = prm.out[2] = prm.out[3] = (__nv_bfloat16*)O;
    prm.status = status;
    CUtensorMap ma[4], mb, mo[4];
    for (int p = 0; p < 4; ++p)
        if (!make_map(&ma[p], As[p < n_a ? p : 0], D, D, N, B * H, kRows))
            return cudaErrorInvalidValue;
    if (!make_map(&mb, W, D, n_a * C, C, 1, (uint32_t)prm.NT) ||
        !make_store_map(&mo[0], O, C, N, B, (uint32_t)D))
        return cudaErrorInvalidValue;
    mo[1] = mo[2] = mo[3] = mo[0];
    switch (D) {
        case 16: return launch<16, 1>(ma, mb, mo, prm, st);
        case 32: return launch<32, 1>(ma, mb, mo, prm, st);
        case 64: return launch<64, 1>(ma, mb, mo, prm, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace flarepp
