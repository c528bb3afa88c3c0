// Tensor-core (tcgen05 / TMEM / TMA) weight-gradient GEMM of the mixer's backward:
//   dW[r][c] = sum over tokens t of A(t, r) B(t, c)
// (dWo = dO^T merge(Y), dW_in = dP^T X, the backward of O = merge(Y) Wo^T and of
// K, V, K~, V~ = X W_in^T in Fig. 1). Both operands are token-major in memory, so the
// contraction runs over tokens with MN-major operand tiles: each tile is a set of D-wide
// channel columns ("atoms") of 64 tokens x D channels each, swizzled to the D-wide row like
// every other operand of the library. A tile arrives as four-dimensional TMA boxes
// {D channels, 64 tokens, atoms, 1} (the atom dimension steps over heads, or over the D-wide
// column blocks of a plain matrix): one box per tile, or one per atom where a tile of a
// HEADS source would cross from one tensor into the next. Few large boxes instead of one
// per atom took dW_in from 1.20 to about 0.3 ms at mesh3d. A channel source is either
//   HEADS: up to four tensors [B*H][N][D] side by side (channel r: tensor r / C, head
//          (r % C) / D, column r % D), or
//   PLAIN: one matrix [B][N][C] (channel r: column r).
// A work item is (128 rows of dW, NT columns of dW, a chunk of one batch element's tokens);
// it writes its float32 partial sum to part[chunk][R][Cc], and a reduce kernel adds the
// chunks in order (deterministic).
//
// Roles (8 warps): warp 0 the TMA producer, warp 1 the MMA issuer, warps 4..7 the epilogue
// (TMEM lane = row of dW). Two TMEM accumulators let the epilogue of one item overlap the
// products of the next. Every wait is bounded (2 s of %globaltimer), as in the other kernels.
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

constexpr int kThreads = 256;
constexpr int kFirstEpiWarp = 4;
constexpr int kRowsW = 128;   // rows of dW per item (TMEM lanes, MMA M)
constexpr int kMaxNT = 256;   // columns of dW per item, at most
constexpr int kTok = 64;      // tokens per pipeline stage (four K = 16 steps)
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint32_t kTmemCols = 512;

template <int D>
struct WCfg {
    static constexpr int kAtom = kTok * D * 2;  // one 64-token x D column, swizzled
    static constexpr int kAStage = (kRowsW / D) * kAtom;
    static constexpr int kBStage = (kMaxNT / D) * kAtom;
    static constexpr int kStage = kAStage + kBStage;
    static constexpr int kStages = (192 * 1024) / kStage > 6 ? 6 : (192 * 1024) / kStage;
    static constexpr uint32_t kSwz = D == 16 ? kSw32 : (D == 32 ? kSw64 : kSw128);
    static constexpr uint32_t kSBO = 8 * D * 2;  // 8-token groups along K
    static constexpr int kNumBars = 2 * kStages + 4 + 1;
    static constexpr int kNeed = 1024 + kStages * kStage + kNumBars * 8 + 16;
    static constexpr int kSmem = kNeed > 122880 ? kNeed : 122880;  // one CTA per SM
    static_assert(kSmem <= 232448, "shared memory budget");
};

struct WgParams {
    int64_t B, N, H, C;
    int64_t R, Cc;         // rows and columns of dW
    int a_heads, b_heads;  // source kinds: 1 = HEADS, 0 = PLAIN
    int a_apb, b_apb;      // atoms per TMA box of each operand
    int NT;
    uint32_t idesc;
    int64_t chunk_len, chunks_per_b, n_chunks;
    int64_t row_tiles, col_tiles, n_items;
    float* part;  // [n_chunks][R][Cc]
    int* status;
};

struct WItem {
    int64_t rt, ct, b, n0, n1, chunk;
};

__device__ __forceinline__ WItem witem(const WgParams& p, int64_t v) {
    WItem w;
    const int64_t tiles = p.row_tiles * p.col_tiles;
    const int64_t t = v % tiles;  // tiles of one chunk run together (their tokens are shared)
    w.chunk = v / tiles;
    w.rt = t / p.col_tiles;
    w.ct = t % p.col_tiles;
    w.b = w.chunk / p.chunks_per_b;
    w.n0 = (w.chunk % p.chunks_per_b) * p.chunk_len;
    w.n1 = min(p.N, w.n0 + p.chunk_len);
    return w;
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

// Load the atoms of channels [c0, c0 + width) of one source for tokens [n0, n0 + kTok) of
// batch element b into consecutive atom slots at dst, in boxes of apb atoms (a box never
// crosses from one tensor of a HEADS source into the next).
template <int D>
__device__ __forceinline__ void load_atoms(uint32_t dst, int heads_kind, const CUtensorMap* m0,
                                           const CUtensorMap* m1, const CUtensorMap* m2,
                                           const CUtensorMap* m3, int64_t c0, int width, int apb,
                                           int64_t C, int64_t b, int n0, uint32_t bar) {
    using W = WCfg<D>;
    for (int k = 0; k < width / (apb * D); ++k) {
        const int64_t c = c0 + (int64_t)k * apb * D;
        const uint32_t d = dst + k * apb * W::kAtom;
        if (heads_kind) {
            const int64_t p = c / C;
            const CUtensorMap* m = p == 0 ? m0 : p == 1 ? m1 : p == 2 ? m2 : m3;
            tma_load_4d(d, m, 0, n0, (int)((c % C) / D), (int)b, bar);
        } else {
            tma_load_4d(d, m0, 0, n0, (int)(c / D), (int)b, bar);
        }
    }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    tc_wgrad_kernel(const __grid_constant__ CUtensorMap tA0, const __grid_constant__ CUtensorMap tA1,
                    const __grid_constant__ CUtensorMap tA2, const __grid_constant__ CUtensorMap tA3,
                    const __grid_constant__ CUtensorMap tB0, const __grid_constant__ CUtensorMap tB1,
                    const __grid_constant__ CUtensorMap tB2, const __grid_constant__ CUtensorMap tB3,
                    const WgParams prm) {
    using W = WCfg<D>;
    constexpr int kS = W::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kS * W::kStage);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + W::kNumBars);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t full0 = smem_u32(bars);
    const uint32_t empty0 = full0 + 8u * kS;
    const uint32_t accfull0 = empty0 + 8u * kS;
    const uint32_t accempty0 = accfull0 + 16u;
    const uint32_t fin = accempty0 + 16u;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int st = 0; st < kS; ++st) {
            mbar_init(full0 + 8u * st, 1);
            mbar_init(empty0 + 8u * st, 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accfull0 + 8u * b, 1);
            mbar_init(accempty0 + 8u * b, kRowsW);
        }
        mbar_init(fin, 1);
        *abort_flag = 0;
        fence_mbar_init();
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
        const uint32_t bytes = (uint32_t)(W::kAStage + (prm.NT / D) * W::kAtom);
        for (int64_t v = blockIdx.x; v < prm.n_items && ok; v += gridDim.x) {
            const WItem I = witem(prm, v);
            for (int64_t n = I.n0; n < I.n1; n += kTok, ++it) {
                const int st = it % kS;
                if (it >= (uint32_t)kS &&
                    !warp_wait(empty0 + 8u * st, ((it / kS) - 1) & 1, abort_flag, prm.status)) {
                    ok = false;
                    break;
                }
                if (elect_one()) {
                    const uint32_t dst = smem_u32(smem + st * W::kStage);
                    mbar_expect_tx(full0 + 8u * st, bytes);
                    load_atoms<D>(dst, prm.a_heads, &tA0, &tA1, &tA2, &tA3, I.rt * kRowsW,
                                  kRowsW, prm.a_apb, prm.C, I.b, (int)n, full0 + 8u * st);
                    load_atoms<D>(dst + W::kAStage, prm.b_heads, &tB0, &tB1, &tB2, &tB3,
                                  I.ct * prm.NT, prm.NT, prm.b_apb, prm.C, I.b, (int)n,
                                  full0 + 8u * st);
                }
                __syncwarp();
            }
        }
        if (!ok) {
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
        for (int64_t v = blockIdx.x; v < prm.n_items && ok; v += gridDim.x, ++j) {
            const WItem I = witem(prm, v);
            const int ab = j & 1;
            if (j >= 2 &&
                !warp_wait(accempty0 + 8u * ab, ((j >> 1) - 1) & 1, abort_flag, prm.status)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t acc = tmem + ab * kMaxNT;
            bool first = true;
            for (int64_t n = I.n0; n < I.n1; n += kTok, ++it) {
                const int st = it % kS;
                if (!warp_wait(full0 + 8u * st, (it / kS) & 1, abort_flag, prm.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a = smem_u32(smem + st * W::kStage);
                const uint32_t b = a + W::kAStage;
#pragma unroll
                for (int k = 0; k < kTok / 16; ++k) {
                    // MN-major operands: K steps of 16 tokens inside each atom; atoms (D-wide
                    // channel columns) kAtom bytes apart along M and N
                    const uint64_t ad = smem_desc(a + k * 16 * D * 2, W::kAtom, W::kSBO, W::kSwz);
                    const uint64_t bd = smem_desc(b + k * 16 * D * 2, W::kAtom, W::kSBO, W::kSwz);
                    if (elect_one()) mma_ss(acc, ad, bd, prm.idesc, (first && k == 0) ? 0u : 1u);
                    __syncwarp();
                }
                first = false;
                if (elect_one()) mma_commit(empty0 + 8u * st);
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
        const int q = warp % 4;
        const int r = 32 * q + lane;
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        uint32_t j = 0;
        for (int64_t v = blockIdx.x; v < prm.n_items; v += gridDim.x, ++j) {
            const WItem I = witem(prm, v);
            const int ab = j & 1;
            if (!warp_wait(accfull0 + 8u * ab, (j >> 1) & 1, abort_flag, prm.status)) break;
            tc_fence_after();
            const uint32_t acc = tmem + lane_off + ab * kMaxNT;
            const int64_t row = I.rt * kRowsW + r;
            float* dst = prm.part + (I.chunk * prm.R + row) * prm.Cc + I.ct * prm.NT;
            for (int c = 0; c < prm.NT; c += 16) {
                uint32_t v16[16];
                tmem_ld16(acc + c, v16);
                tmem_wait_ld16(v16);
                if (row < prm.R) {
                    float4* d4 = reinterpret_cast<float4*>(dst + c);
#pragma unroll
                    for (int g = 0; g < 4; ++g)
                        d4[g] = make_float4(__uint_as_float(v16[4 * g]), __uint_as_float(v16[4 * g + 1]),
                                            __uint_as_float(v16[4 * g + 2]),
                                            __uint_as_float(v16[4 * g + 3]));
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

// dW = sum of the chunks' partials, in chunk order; rows r < R_out take the sum of the rows
// r + k * R_out for k < fold (fold 2 adds the gradients of tied projections).
__global__ void wgrad_reduce_kernel(const float* __restrict__ part, int64_t n_chunks, int64_t R,
                                    int64_t Cc, int64_t R_out, int fold,
                                    __nv_bfloat16* __restrict__ out) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= R_out * Cc) return;
    const int64_t r = i / Cc, c = i % Cc;
    float acc = 0.f;
    for (int k = 0; k < fold; ++k)
        for (int64_t ch = 0; ch < n_chunks; ++ch) acc += part[(ch * R + r + k * R_out) * Cc + c];
    out[i] = __float2bfloat16_rn(acc);
}

__global__ void transpose_bf16_kernel(const __nv_bfloat16* __restrict__ src, int64_t R,
                                      int64_t Cc, int rep, __nv_bfloat16* __restrict__ dst) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;  // index into dst
    const int64_t cols = rep * R;
    if (i >= Cc * cols) return;
    const int64_t c = i / cols, j = i % cols;
    dst[i] = src[(j % R) * Cc + c];
}

__global__ void add_bf16_kernel(__nv_bfloat16* __restrict__ dst,
                                const __nv_bfloat16* __restrict__ src, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = __float2bfloat16_rn(__bfloat162float(dst[i]) + __bfloat162float(src[i]));
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

// bf16 {D channels, N tokens, atoms, B} with the given byte strides of dimensions 1..3;
// boxes of D x kTok x `atoms` x 1, swizzled to the D-wide row. In shared memory a box is
// atom-major: atom a is the kTok x D block at a * kTok * D * 2.
bool make_map(CUtensorMap* m, const void* base, int64_t D, int64_t N, int64_t n_atoms,
              int64_t B, int64_t s_tok, int64_t s_atom, int64_t s_b, int atoms) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)N, (cuuint64_t)n_atoms, (cuuint64_t)B};
    cuuint64_t strides[3] = {(cuuint64_t)s_tok, (cuuint64_t)s_atom, (cuuint64_t)s_b};
    cuuint32_t box[4] = {(cuuint32_t)D, (cuuint32_t)kTok, (cuuint32_t)atoms, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    const CUtensorMapSwizzle sw = D == 16 ? CU_TENSOR_MAP_SWIZZLE_32B
                                          : (D == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                     : CU_TENSOR_MAP_SWIZZLE_128B);
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Atoms per box for tiles of `width` channels: the whole tile, unless a tile of a HEADS
// source could cross from one tensor into the next (C not a multiple of the width).
int atoms_per_box(const WgradSource& s, int64_t C, int64_t D, int width) {
    return (s.heads && C % width != 0) ? 1 : width / (int)D;
}

// the maps of one source, for boxes of `atoms` atoms: HEADS (n tensors [B*H][N][D], the
// atoms are heads) or PLAIN ([B][N][C], the atoms are the D-wide column blocks)
bool source_maps(CUtensorMap* m, const WgradSource& s, int64_t B, int64_t N, int64_t H,
                 int64_t D, int atoms) {
    for (int p = 0; p < 4; ++p) {
        const void* base = s.t[p < s.n ? p : 0];
        const bool ok = s.heads ? make_map(&m[p], base, D, N, H, B, D * 2, N * D * 2,
                                           H * N * D * 2, atoms)
                                : make_map(&m[p], base, D, N, H, B, H * D * 2, D * 2,
                                           N * H * D * 2, atoms);
        if (!ok) return false;
    }
    return true;
}

template <int D>
cudaError_t launch(const CUtensorMap* ma, const CUtensorMap* mb, const WgParams& prm,
                   cudaStream_t st) {
    using Wc = WCfg<D>;
    const cudaError_t attr = ensure_smem_limit((const void*)tc_wgrad_kernel<D>, Wc::kSmem);
    if (attr != cudaSuccess) return attr;
    if (prm.n_items == 0) return cudaSuccess;
    int dev = 0, sms = kNumSMs;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t grid = prm.n_items < sms ? prm.n_items : sms;
    tc_wgrad_kernel<D><<<(unsigned)grid, kThreads, Wc::kSmem, st>>>(
        ma[0], ma[1], ma[2], ma[3], mb[0], mb[1], mb[2], mb[3], prm);
    return cudaGetLastError();
}

}  // namespace

cudaError_t transpose_bf16(const void* src, int64_t R, int64_t Cc, int rep, void* dst,
                           cudaStream_t st) {
    const int64_t n = Cc * rep * R;
    if (n == 0) return cudaSuccess;
    transpose_bf16_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(
        (const __nv_bfloat16*)src, R, Cc, rep, (__nv_bfloat16*)dst);
    return cudaGetLastError();
}

cudaError_t add_bf16(void* dst, const void* src, int64_t n, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const int64_t blocks = (n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096;
    add_bf16_kernel<<<(unsigned)blocks, 256, 0, st>>>((__nv_bfloat16*)dst,
                                                      (const __nv_bfloat16*)src, n);
    return cudaGetLastError();
}

WgradPlan wgrad_plan(int64_t B, int64_t N, int64_t R, int64_t Cc) {
    WgradPlan w{};
    int nt = kMaxNT;
    while (nt > 16 && Cc % nt != 0) nt /= 2;
    w.NT = nt;
    w.row_tiles = (R + kRowsW - 1) / kRowsW;
    w.col_tiles = Cc / nt;
    // about four items per SM, chunks of whole 64-token stages inside one batch element
    const int64_t tiles = w.row_tiles * w.col_tiles;
    int64_t want = (4 * kNumSMs + tiles - 1) / tiles;
    int64_t per_b = (want + B - 1) / B;
    if (per_b < 1) per_b = 1;
    w.chunk_len = ((N + per_b - 1) / per_b + kTok - 1) / kTok * kTok;
    if (w.chunk_len < kTok) w.chunk_len = kTok;
    w.chunks_per_b = (N + w.chunk_len - 1) / w.chunk_len;
    w.n_chunks = B * w.chunks_per_b;
    w.part_bytes = (size_t)w.n_chunks * (size_t)R * (size_t)Cc * sizeof(float);
    return w;
}

cudaError_t tc_wgrad(int64_t B, int64_t N, int64_t H, int64_t D, const WgradSource& a,
                     const WgradSource& b, int64_t R, int64_t Cc, int64_t R_out, int fold,
                     float* part, void* dW, int* status, cudaStream_t st) {
    const WgradPlan w = wgrad_plan(B, N, R, Cc);
    if (w.NT % D != 0 || R % D != 0) return cudaErrorInvalidValue;
    WgParams prm{};
    prm.B = B;
    prm.N = N;
    prm.H = H;
    prm.C = H * D;
    prm.R = R;
    prm.Cc = Cc;
    prm.a_heads = a.heads;
    prm.b_heads = b.heads;
    prm.NT = w.NT;
    prm.idesc = idesc_bf16_f32(kRowsW, w.NT, true, true);
    prm.chunk_len = w.chunk_len;
    prm.chunks_per_b = w.chunks_per_b;
    prm.n_chunks = w.n_chunks;
    prm.row_tiles = w.row_tiles;
    prm.col_tiles = w.col_tiles;
    prm.n_items = w.n_chunks * w.row_tiles * w.col_tiles;
    prm.part = part;
    prm.status = status;
    CUtensorMap ma[4], mb[4];
    prm.a_apb = atoms_per_box(a, H * D, D, kRowsW);
    prm.b_apb = atoms_per_box(b, H * D, D, w.NT);
    if (!source_maps(ma, a, B, N, H, D, prm.a_apb) || !source_maps(mb, b, B, N, H, D, prm.b_apb))
        return cudaErrorInvalidValue;
    cudaError_t e;
    switch (D) {
        case 16: e = launch<16>(ma, mb, prm, st); break;
        case 32: e = launch<32>(ma, mb, prm, st); break;
        case 64: e = launch<64>(ma, mb, prm, st); break;
        default: return cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
    const int64_t n = R_out * Cc;
    wgrad_reduce_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(
        part, w.n_chunks, R, Cc, R_out, fold, (__nv_bfloat16*)dW);
    return cudaGetLastError();
}

}  // namespace flarepp
