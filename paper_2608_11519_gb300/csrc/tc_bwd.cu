// Tensor-core (tcgen05 / TMEM / TMA) backward of the routing chain, bf16 inputs (App. A.5).
//
// Every SDPA(A, B, C) of the chain is differentiated from its saved log-normaliser L
// (base 2) and c = <dO, O>:  P = 2^(x - L) with x = scale log2(e) <a, b>,
// dS = P o (dP - c) with dP = <dO, C>, and the products dA = s dS B, dB = s dS^T A,
// dC = P^T dO. Five passes cover the three calls (T23 in one of two forms). In every pass a
// score tile of 128 TMEM lanes x kItem columns is produced by the tensor cores, turned into
// bf16 P and dS in place by a softmax warpgroup, and consumed as the TMEM A operand of one or
// two accumulating products whose B operand is the same streamed item:
//
//   route-row passes (TMEM lanes are routes, items are tokens; per-chunk partial sums):
//     R3  call 3, column statistics L3, c3 of the tokens:
//         S = Q K^T, dP = Z dY^T;  acc0 += dS K (-> dQ / s),  acc1 += P dY (-> dZ)
//     R2  call 2, row statistics L2, c2:   S = Q K^T,  dP = dZ V^T;   acc0 += dS K
//     R1  call 1, row statistics L1, c1:   S = Qs Kt^T, dP = dQ Vt^T; acc0 += dS Kt
//   token-row passes (TMEM lanes are tokens, items are routes; final per-token outputs):
//     T23 calls 3 and 2, token statistics L3, c3 and route statistics L2, c2:
//         S = K Q^T, dP2 = V dZ^T, dP3 = dY Z^T,
//         dS = P2 o (dP2 - c2) + P3 o (dP3 - c3) with P2 = 2^(x - L2), P3 = 2^(x - L3);
//         acc0 += dS Q (-> dK / s),  acc1 += P2 dZ (-> dV)
//     T1  call 1, route statistics L1, c1:  S = Kt Qs^T, dP = Vt dQ^T;
//         acc0 += dS Qs (-> dKt / s),  acc1 += P dQ (-> dVt)
//     T23C  T23 with its two dP products merged into one of depth 2D (see slice_math),
//         one exponential per score and its A tiles in TMEM; it serves every (b, h) whose
//         statistics allow it (D = 16, 32), T23 the others
// Score products take both operands from shared memory (TMA, swizzled, K-major), except in
// T23C (A from TMEM); the accumulating products read P or dS from TMEM and the item,
// MN-major, from shared memory.
//
// Roles: one MMA warp per TMEM stream of 128 rows (a commit stalls only the warp that
// issues it), one softmax warpgroup per stream (warps 4..), and a TMA producer warp that
// also stages each item's column statistics in shared memory. A pass has as many streams as
// its TMEM columns allow (at most four), with the widest item (64, 48 or 32 rows) that fits
// that count (T23 and T23C: two streams of 64 rows); the softmax works on 16-column slices
// in packed f32x2 arithmetic. A work unit is (b*h, group of NS x 128 rows, chunk of items).
// Every wait is bounded (2 s of %globaltimer): on expiry the kernel records
// FLAREPP_ERR_TIMEOUT in the status word, every role leaves its loops, the producer waits
// for its copies in flight, the MMA issuer for its products, and TMEM is freed.
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

constexpr int kFirstSoftmaxWarp = 4;
constexpr int kRows = 128;  // TMEM lanes per stream, MMA M

constexpr uint32_t kTmemCols = 512;

enum Pass : int { kR3 = 0, kR2 = 1, kR1 = 2, kT23 = 3, kT1 = 4, kT23C = 5 };

// LO (D <= 32; the backward of the training forward, whose calls 2 and 3 take Q as a hi/lo
// pair of bf16 operands): the score products S = Q K^T (R3, R2) and S = K Q^T (T23, T23C) add
// the product with Q's lo tile, kept as one more A tile (R3, R2) or item tile (T23, T23C)
// after the others. Nothing else changes: the TMEM layout, items and statistics are LO's too.
template <int D, int PASS, bool LO = false>
struct BCfg {
    static_assert(!LO || D <= 32, "the hi/lo form of Q serves D = 16 and 32");
    static constexpr bool kRouteRows = PASS <= kR1;
    // T23C (calls 3 and 2 with their two dP products merged into one, see bwd_slice) keeps
    // its A tiles in TMEM and multiplies them from there (`ts` products)
    static constexpr bool kATmem = PASS == kT23C;
    static constexpr int kNA = PASS == kT23 ? 3 : 2;  // score products (TMEM score tiles)
    static constexpr int kNT = (PASS == kT23 || PASS == kT23C) ? 3 : 2;  // A and item tiles
    static constexpr int kNAcc = (PASS == kR2 || PASS == kR1) ? 1 : 2;
    static constexpr bool kLoA = LO && (PASS == kR3 || PASS == kR2);   // Q is A operand 0
    static constexpr bool kLoI = LO && (PASS == kT23 || PASS == kT23C);  // Q is item operand 0
    static constexpr int kNTA = kNT + (kLoA ? 1 : 0);  // A tiles per stream in shared memory
    static constexpr int kNTI = kNT + (kLoI ? 1 : 0);  // item tiles per ring stage
    static constexpr bool kColStats = PASS == kR3 || PASS == kT23 || PASS == kT1 || kATmem;
    static constexpr bool kRowStats = PASS == kR2 || PASS == kR1 || PASS == kT23 || kATmem;
    // TMEM per stream: kNA score tiles of kItem columns, kNAcc accumulators of D, then (T23C)
    // the kNT bf16 A tiles of D / 2 columns, padded to 32 columns. The most streams (at most four) that fit in 512
    // columns, with the widest item of 64, 48 or 32 rows for that count: four streams make a
    // 512-row group, so M = 512 fills every unit.
    static constexpr uint32_t col_stream(int item) {
        return kATmem ? (kNA * item + kNAcc * D + kNT * D / 2 + 31) / 32 * 32
                      : kNA * item + kNAcc * D;
    }
    static constexpr int fits(int ns, int item) { return ns * col_stream(item) <= kTmemCols; }
    static constexpr int pick_ns() {
        // T23 (three score products, 6 ss MMAs per item): two streams of 64-row items
        // measured faster than three of 32 (3.41 vs 3.60 ms at mesh3d); for R3 and T1 the
        // most streams win (two of 64 rows: 3.67 vs 2.12 ms; three of 48: 2.38 vs 2.17 ms)
        if ((PASS == kT23 || PASS == kT23C) && fits(2, 64)) return 2;
        for (int ns = 4; ns >= 1; --ns)
            if (fits(ns, 32)) return ns;
        return 0;
    }
    static constexpr int NS = pick_ns();
    static_assert(NS >= 1, "TMEM budget");
    static constexpr int kItem = fits(NS, 64) ? 64 : (fits(NS, 48) ? 48 : 32);
    static constexpr uint32_t kColStream = col_stream(kItem);
    // warps 0..NS-1 issue MMAs (one per stream), warps 4.. are the softmax warpgroups, and
    // the TMA producer is warp 3 (NS < 4) or the warp after the softmax warps (NS = 4)
    static constexpr int kProdWarp = NS < 4 ? 3 : kFirstSoftmaxWarp + 4 * NS;
    static constexpr int kWarps = kFirstSoftmaxWarp + 4 * NS + (NS < 4 ? 0 : 1);
    static constexpr int kThreads = kWarps * 32;
    static constexpr int kGroup = NS * kRows;  // rows per work unit
    static constexpr int kStages = kItem == 64 ? 6 : 10;
    static constexpr int kATile = kRows * D * 2;
    static constexpr int kABytes = NS * kNTA * kATile;  // one unit's A tiles
    static constexpr int kItemTile = kItem * D * 2;
    static constexpr int kStage = kNTI * kItemTile;
    // two shared-memory copies of a unit's A tiles when they fit beside the ring
    static constexpr int kABuf = 2 * kABytes + kStages * kStage <= 200 * 1024 ? 2 : 1;
    static constexpr uint32_t kSwz = D == 16 ? kSw32 : (D == 32 ? kSw64 : kSw128);
    static constexpr uint32_t kSBO = 8 * D * 2;
    // barriers: full[S], empty[S], afull[kABuf], afree[kABuf], then per stream sready,
    //           pready, accdone, accfree, fin, aready (T23C: the A tiles are in TMEM)
    static constexpr int kNumBars = 2 * kStages + 2 * kABuf + 6 * NS;
    static constexpr int kStatBytes = kStages * 2 * kItem * 4;
    static constexpr int kData = kABuf * kABytes + kStages * kStage;
    static constexpr int kNeed = 1024 + kData + kStatBytes + kNumBars * 8 + 16;
    // at least 120 KB so that one CTA owns an SM and its 512 TMEM columns
    static constexpr int kSmem = kNeed > 122880 ? kNeed : 122880;
    static_assert(kSmem <= 232448, "shared memory budget");
    static constexpr uint32_t kIdescS = idesc_bf16_f32(128, kItem, false, false);
    static constexpr uint32_t kIdescAcc = idesc_bf16_f32(128, D, false, true);
    static constexpr uint32_t kColA = kNA * kItem + kNAcc * D;  // T23C: first A column
    static_assert(!kATmem || D <= 32, "T23C serves D = 16 and 32");
};

struct BwdParams {
    int64_t BH, H, N, M;
    float c;      // scale * log2(e), signed
    float scale;  // s
    int a0_per_head;            // R1: the first A operand (seeds) is indexed by head
    int i0_per_head;            // T1: the first item operand (seeds) is indexed by head
    int64_t chunk_len, nchunk;  // route-row passes
    int64_t n_groups;           // route groups (route-row passes) or token groups
    int64_t n_units;
    const float* Lrow;  // row statistics [BH][rows]: L (base 2) and c
    const float* crow;
    const float* Lcol;  // column statistics [BH][items' rows]
    const float* ccol;
    float* pa;  // route-row passes: partial sums [BH][nchunk][M][D] (acc1, acc0)
    float* pb;
    __nv_bfloat16* out0;  // token-row passes: s * acc0 and acc1, [BH][N][D]
    __nv_bfloat16* out1;
    const float* Rb;    // T23C: the shift R of each (b, h) [BH]
    const int* flags;   // when not null: only the units of (b, h) with flags[bh] == want run
    int want;
    int* status;
    uint64_t wait_ns;     // bound of every wait (2 s unless the test hook is set)
    int64_t withhold_it;  // test hook: ring item of CTA 0 the producer never loads (-1: none)
};

// Units of a (b, h) whose flag differs from the one this launch serves are skipped by every
// role alike (no barrier, copy or product is issued for them).
__device__ __forceinline__ bool unit_skipped(const BwdParams& p, int64_t bh) {
    return p.flags != nullptr && p.flags[bh] != p.want;
}
// The unit before this CTA's first unit of the next (b, h): units are numbered (b, h)-major
// with per_bh units each, and a CTA takes every gridDim.x-th one, so a skipped (b, h) is
// stepped over whole.
__device__ __forceinline__ int64_t skip_bh(int64_t bh, int64_t per_bh) {
    const int64_t next = (bh + 1) * per_bh;
    const int64_t g = gridDim.x;
    return next + ((int64_t)blockIdx.x - next % g + g) % g - g;
}

struct BUnit {
    int64_t bh, g, chunk;
    int64_t row0;  // first TMEM row (route or token) of stream 0
    int64_t rows;  // route or token count of the rows' dimension (M or N)
    int64_t item0, item_end;
    int n_act;  // streams with at least one valid row
    int n_items;
};

template <int D, int PASS>
__device__ __forceinline__ BUnit bwd_unit(const BwdParams& p, int64_t u) {
    using C = BCfg<D, PASS>;
    BUnit U;
    if (C::kRouteRows) {
        U.chunk = u % p.nchunk;
        const int64_t t = u / p.nchunk;
        U.g = t % p.n_groups;
        U.bh = t / p.n_groups;
        U.rows = p.M;
        U.item0 = U.chunk * p.chunk_len;
        U.item_end = min(p.N, U.item0 + p.chunk_len);
    } else {
        U.g = u % p.n_groups;
        U.bh = u / p.n_groups;
        U.chunk = 0;
        U.rows = p.N;
        U.item0 = 0;
        U.item_end = p.M;
    }
    U.row0 = U.g * C::kGroup;
    const int64_t left = U.rows - U.row0;
    U.n_act = left >= C::kGroup ? C::NS : (int)((left + kRows - 1) / kRows);
    U.n_items = (int)((U.item_end - U.item0 + C::kItem - 1) / C::kItem);
    return U;
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

// packed pairs of f32 (lo, hi) in one 64-bit register
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
    uint64_t d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b) {
    uint64_t d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ uint64_t ex2x2(uint64_t x) {
    float a, b;
    unpack_f32x2(x, a, b);
    return pack_f32x2(ex2(a), ex2(b));
}
// bf16 pair (lo in the low half) from a packed f32 pair
__device__ __forceinline__ uint32_t bf16x2(uint64_t v) {
    uint32_t r;
    asm("{\n\t.reg .f32 a, b;\n\tmov.b64 {a, b}, %1;\n\tcvt.rn.bf16x2.f32 %0, b, a;\n\t}"
        : "=r"(r)
        : "l"(v));
    return r;
}
__device__ __forceinline__ uint64_t ld_pair(const uint32_t* r, int k) {
    return pack_f32x2(__uint_as_float(r[2 * k]), __uint_as_float(r[2 * k + 1]));
}

// Bounded wait on an mbarrier phase. Returns false when the kernel is aborting.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                         int* status, uint64_t limit) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 63u) == 0) {
            if (*abort_flag) return false;
            if (globaltimer_ns() - t0 > limit) {
                *abort_flag = 1;
                atomicExch(status, (int)FLAREPP_ERR_TIMEOUT);
                return false;
            }
        }
    }
}
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          int* status, uint64_t limit) {
    const bool got = wait_bar(bar, parity, abort_flag, status, limit);
    return __all_sync(0xffffffffu, got);
}

// One 16-column slice h of an item for this thread's row (slice_load, slice_wait,
// slice_math): reads the score tiles, writes bf16 dS over score tile 0 and (when a second
// accumulator reads it) bf16 P over score tile 1. Math on packed f32 pairs. The row
// statistics come as (-L, -L) and (-c, -c) pairs; the column statistics sit negated in
// shared memory. When the item is short (FULL false), columns at or beyond nv get
// P = dS = 0.
//
// T23C merges the two dP products of T23. With r = P2 / P3 = 2^(L3[n] - L2[m]) = u[n] w[m],
// u[n] = 2^(L3[n] - R), w[m] = 2^(R - L2[m]) for a shift R per (b, h), score tile 1 holds
//   T = dP3 + r dP2 = [dY | u V] [Z | w dZ]^T   (one product of depth 2D),
// so that dS = P2 (dP2 - c2) + P3 (dP3 - c3) = P3 (T - c3 - u (w c2)), and E2 = P3 u =
// 2^(c x - R) = P2 / w goes to tile 1: the second accumulator multiplies it by w dZ, giving
// P2 dZ. One exponential per score. The column statistic is -(w c2); u2 holds (u, u).
// (Where P3 underflows, P2 = P3 u w stays below 2^-66: R bounds u by 2^60 and w by 1.)
template <int D, int PASS>
struct SliceRegs {
    uint32_t sr[16], d1[16], d2[PASS == kT23 ? 16 : 1];
};
template <int D, int PASS>
__device__ __forceinline__ void slice_load(uint32_t t0, int h, SliceRegs<D, PASS>& g) {
    using C = BCfg<D, PASS>;
    tmem_ld16(t0 + 16 * h, g.sr);
    tmem_ld16(t0 + C::kItem + 16 * h, g.d1);
    if (PASS == kT23) tmem_ld16(t0 + 2 * C::kItem + 16 * h, g.d2);
}
template <int D, int PASS>
__device__ __forceinline__ void slice_wait(SliceRegs<D, PASS>& g) {
    tmem_wait_ld16(g.sr);
    tmem_wait_ld16(g.d1);
    if (PASS == kT23) tmem_wait_ld16(g.d2);
}
template <int D, int PASS, bool FULL>
__device__ __forceinline__ void slice_math(uint32_t t0, int h, const SliceRegs<D, PASS>& g, int nv,
                                           uint64_t c2, uint64_t nLr2, uint64_t ncr2,
                                           const float* nLc, const float* ncc, uint64_t u2) {
    using C = BCfg<D, PASS>;
    uint32_t ds[8], pp[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const int col = 16 * h + 2 * k;
        const uint64_t x = ld_pair(g.sr, k);
        const uint64_t dp = ld_pair(g.d1, k);
        uint64_t p, d;
        if (PASS == kR2 || PASS == kR1) {
            p = ex2x2(fma2(x, c2, nLr2));
            d = mul2(p, add2(dp, ncr2));
        } else if (PASS == kT23C) {
            const uint64_t nwc = *reinterpret_cast<const uint64_t*>(nLc + col);
            const uint64_t p3 = ex2x2(fma2(x, c2, nLr2));
            p = mul2(p3, u2);  // E2 = P3 u
            d = mul2(p3, fma2(u2, nwc, add2(dp, ncr2)));
        } else {
            const uint64_t nL = *reinterpret_cast<const uint64_t*>(nLc + col);
            const uint64_t nc = *reinterpret_cast<const uint64_t*>(ncc + col);
            p = ex2x2(fma2(x, c2, nL));
            d = mul2(p, add2(dp, nc));
            if (PASS == kT23) {
                const uint64_t p3 = ex2x2(fma2(x, c2, nLr2));
                d = fma2(p3, add2(ld_pair(g.d2, k), ncr2), d);
            }
        }
        if (!FULL) {
            float a, b;
            unpack_f32x2(d, a, b);
            d = pack_f32x2(col < nv ? a : 0.f, col + 1 < nv ? b : 0.f);
            unpack_f32x2(p, a, b);
            p = pack_f32x2(col < nv ? a : 0.f, col + 1 < nv ? b : 0.f);
        }
        ds[k] = bf16x2(d);
        pp[k] = bf16x2(p);
    }
    tmem_st8(t0 + 8 * h, ds);
    if (C::kNAcc == 2) tmem_st8(t0 + C::kItem + 8 * h, pp);
}

// One item for this thread's row, 16 columns at a time. (Issuing the next slice's loads
// before the current slice's math measured slower in every pass.)
template <int D, int PASS, bool FULL>
__device__ __forceinline__ void bwd_item(uint32_t t0, int nv, uint64_t c2, uint64_t nLr2,
                                         uint64_t ncr2, const float* nLc, const float* ncc,
                                         uint64_t u2) {
    using C = BCfg<D, PASS>;
#pragma unroll
    for (int h = 0; h < C::kItem / 16; ++h) {
        SliceRegs<D, PASS> g;
        slice_load<D, PASS>(t0, h, g);
        slice_wait<D, PASS>(g);
        slice_math<D, PASS, FULL>(t0, h, g, nv, c2, nLr2, ncr2, nLc, ncc, u2);
    }
}

// ------------------------------------------------------------------ the kernel

template <int D, int PASS, bool LO>
__global__ void __launch_bounds__(BCfg<D, PASS>::kThreads, 1)
    tc_bwd_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
                  const __grid_constant__ CUtensorMap tmA2, const __grid_constant__ CUtensorMap tmI0,
                  const __grid_constant__ CUtensorMap tmI1, const __grid_constant__ CUtensorMap tmI2,
                  const __grid_constant__ CUtensorMap tmLo, const BwdParams prm) {
    using C = BCfg<D, PASS, LO>;
    constexpr int NS = C::NS;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    uint8_t* abuf = smem;                          // kABuf x [NS][kNTA] A tiles
    uint8_t* ring = smem + C::kABuf * C::kABytes;  // kStages x kNTI item tiles, swizzled
    float* stats = reinterpret_cast<float*>(ring + C::kStages * C::kStage);  // [S][2][kItem]
    uint64_t* bars = reinterpret_cast<uint64_t*>(stats + C::kStages * 2 * C::kItem);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::kNumBars);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const uint32_t full0 = smem_u32(bars);
    const uint32_t empty0 = full0 + 8u * C::kStages;
    const uint32_t afull0 = empty0 + 8u * C::kStages;
    const uint32_t afree0 = afull0 + 8u * C::kABuf;
    const uint32_t sready0 = afree0 + 8u * C::kABuf;
    const uint32_t pready0 = sready0 + 8u * NS;
    const uint32_t accdone0 = pready0 + 8u * NS;
    const uint32_t accfree0 = accdone0 + 8u * NS;
    const uint32_t fin0 = accfree0 + 8u * NS;
    const uint32_t aready0 = fin0 + 8u * NS;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int st = 0; st < C::kStages; ++st) {
            mbar_init(full0 + 8u * st, C::kColStats ? 33 : 1);
            mbar_init(empty0 + 8u * st, NS);
        }
        for (int b = 0; b < C::kABuf; ++b) {
            mbar_init(afull0 + 8u * b, 1);
            // released by each stream's MMA warp, or (A in TMEM) by every softmax thread
            // once its rows are copied
            mbar_init(afree0 + 8u * b, C::kATmem ? NS * kRows : NS);
        }
        for (int s = 0; s < NS; ++s) {
            mbar_init(sready0 + 8u * s, 1);
            mbar_init(pready0 + 8u * s, kRows);
            mbar_init(accdone0 + 8u * s, 1);
            mbar_init(accfree0 + 8u * s, kRows);
            mbar_init(fin0 + 8u * s, 1);
            mbar_init(aready0 + 8u * s, kRows);
        }
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmA0);
        prefetch_tmap(&tmA1);
        prefetch_tmap(&tmI0);
        prefetch_tmap(&tmI1);
        if (C::kNT == 3) {
            prefetch_tmap(&tmA2);
            prefetch_tmap(&tmI2);
        }
        if (LO) prefetch_tmap(&tmLo);
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == C::kProdWarp) {
        // ------------------------------------------------------------ TMA producer
        uint32_t it = 0, ua = 0, a_issued = 0;
        int64_t withheld = -1;
        bool ok = true;
        for (int64_t u = blockIdx.x; u < prm.n_units && ok; u += gridDim.x) {
            const BUnit U = bwd_unit<D, PASS>(prm, u);
            if (unit_skipped(prm, U.bh)) {
                u = skip_bh(U.bh, C::kRouteRows ? prm.n_groups * prm.nchunk : prm.n_groups);
                continue;
            }
            const uint32_t uc = ua++;
            const int ab = uc % C::kABuf;
            if (uc >= (uint32_t)C::kABuf &&
                !warp_wait(afree0 + 8u * ab, ((uc / C::kABuf) - 1) & 1, abort_flag, prm.status, prm.wait_ns)) {
                ok = false;
                break;
            }
            if (elect_one()) {
                mbar_expect_tx(afull0 + 8u * ab, U.n_act * C::kNTA * C::kATile);
                const int za0 = (int)(prm.a0_per_head ? U.bh % prm.H : U.bh);
                for (int s = 0; s < U.n_act; ++s) {
                    const int row = (int)(U.row0 + s * kRows);
                    uint8_t* dst = abuf + ab * C::kABytes + s * C::kNTA * C::kATile;
                    tma_load_3d(smem_u32(dst), &tmA0, 0, row, za0, afull0 + 8u * ab);
                    tma_load_3d(smem_u32(dst + C::kATile), &tmA1, 0, row, (int)U.bh,
                                afull0 + 8u * ab);
                    if (C::kNT == 3)
                        tma_load_3d(smem_u32(dst + 2 * C::kATile), &tmA2, 0, row, (int)U.bh,
                                    afull0 + 8u * ab);
                    if (C::kLoA)
                        tma_load_3d(smem_u32(dst + C::kNT * C::kATile), &tmLo, 0, row, (int)U.bh,
                                    afull0 + 8u * ab);
                }
            }
            __syncwarp();
            ++a_issued;
            const int zi0 = (int)(prm.i0_per_head ? U.bh % prm.H : U.bh);
            const float R = C::kATmem ? prm.Rb[U.bh] : 0.f;
            for (int i = 0; i < U.n_items; ++i, ++it) {
                const int st = it % C::kStages;
                if (it >= (uint32_t)C::kStages &&
                    !warp_wait(empty0 + 8u * st, ((it / C::kStages) - 1) & 1, abort_flag,
                               prm.status, prm.wait_ns)) {
                    ok = false;
                    break;
                }
                if (blockIdx.x == 0 && (int64_t)it == prm.withhold_it) {
                    withheld = it;  // never loaded: the waits of its consumers run out
                    continue;
                }
                const int64_t row = U.item0 + (int64_t)i * C::kItem;
                if (elect_one()) {
                    mbar_expect_tx(full0 + 8u * st, C::kStage);
                    const uint32_t dst = smem_u32(ring + st * C::kStage);
                    tma_load_3d(dst, &tmI0, 0, (int)row, zi0, full0 + 8u * st);
                    tma_load_3d(dst + C::kItemTile, &tmI1, 0, (int)row, (int)U.bh,
                                full0 + 8u * st);
                    if (C::kNT == 3)
                        tma_load_3d(dst + 2 * C::kItemTile, &tmI2, 0, (int)row, (int)U.bh,
                                    full0 + 8u * st);
                    if (C::kLoI)
                        tma_load_3d(dst + C::kNT * C::kItemTile, &tmLo, 0, (int)row, (int)U.bh,
                                    full0 + 8u * st);
                    // streams idle in this unit count as having released the stage
                    for (int x = U.n_act; x < NS; ++x) mbar_arrive(empty0 + 8u * st);
                }
                __syncwarp();
                if (C::kColStats) {
                    // the item's column statistics, negated (P = 2^(c x + (-L))); T23C
                    // stages -(w c2) with w = 2^(R - L2)
                    float* sl = stats + st * 2 * C::kItem;
                    const int64_t nvalid = U.item_end - row;
                    for (int k = lane; k < C::kItem; k += 32) {
                        const bool in = k < nvalid;
                        const int64_t idx = U.bh * (C::kRouteRows ? prm.N : prm.M) + row + k;
                        if (C::kATmem) {
                            sl[k] = in ? -exp2f(R - prm.Lcol[idx]) * prm.ccol[idx] : 0.f;
                        } else {
                            sl[k] = in ? -prm.Lcol[idx] : 0.f;
                            sl[C::kItem + k] = in ? -prm.ccol[idx] : 0.f;
                        }
                    }
                    mbar_arrive(full0 + 8u * st);
                }
            }
        }
        // after an abort: wait (bounded) until the newest copy of every buffer has landed
        if (!ok) {
            const uint64_t t0 = globaltimer_ns();
            for (int st = 0; st < C::kStages && (uint32_t)st < it; ++st) {
                const uint32_t x = it - 1 - ((it - 1 - st) % C::kStages);
                while ((int64_t)x != withheld &&
                       !mbar_try_wait(full0 + 8u * st, (x / C::kStages) & 1) &&
                       globaltimer_ns() - t0 < prm.wait_ns) {
                }
            }
            for (int b = 0; b < C::kABuf && (uint32_t)b < a_issued; ++b) {
                const uint32_t x = a_issued - 1 - ((a_issued - 1 - b) % C::kABuf);
                while (!mbar_try_wait(afull0 + 8u * b, (x / C::kABuf) & 1) &&
                       globaltimer_ns() - t0 < prm.wait_ns) {
                }
            }
        }
    } else if (warp < NS) {
        // ------------------------------------------------------------ MMA warp of stream s
        // For item j: the accumulating products of item j - 1 (after its P / dS is written)
        // and the score products of item j, then one commit that the softmax waits on. The
        // softmax frees ring stage j - 1 once S(j) is complete (the tensor pipe runs this
        // warp's products in order), and the last stage of a unit after acc_done.
        const int s = warp;
        uint32_t it = 0, ua = 0, pj = 0, nu = 0, ar = 0;
        bool ok = true;
        auto wait = [&](uint32_t bar, uint32_t parity) {
            return warp_wait(bar, parity, abort_flag, prm.status, prm.wait_ns);
        };
        const uint32_t t0 = tmem + s * C::kColStream;
        const uint32_t acc = t0 + C::kNA * C::kItem;
        auto issue_acc = [&](int stg, bool accumulate) {
            const uint32_t ib = smem_u32(ring + stg * C::kStage);
#pragma unroll
            for (int k = 0; k < C::kItem / 16; ++k) {
                const uint64_t bd = smem_desc(ib + k * 16 * D * 2, C::kItemTile, C::kSBO, C::kSwz);
                if (elect_one())
                    mma_ts(acc, t0 + 8 * k, bd, C::kIdescAcc, (accumulate || k > 0) ? 1u : 0u);
                __syncwarp();
            }
            if (C::kNAcc == 2) {
#pragma unroll
                for (int k = 0; k < C::kItem / 16; ++k) {
                    const uint64_t bd = smem_desc(ib + C::kItemTile + k * 16 * D * 2, C::kItemTile,
                                                  C::kSBO, C::kSwz);
                    if (elect_one())
                        mma_ts(acc + D, t0 + C::kItem + 8 * k, bd, C::kIdescAcc,
                               (accumulate || k > 0) ? 1u : 0u);
                    __syncwarp();
                }
            }
        };
        for (int64_t u = blockIdx.x; u < prm.n_units && ok; u += gridDim.x) {
            const BUnit U = bwd_unit<D, PASS>(prm, u);
            if (unit_skipped(prm, U.bh)) {
                u = skip_bh(U.bh, C::kRouteRows ? prm.n_groups * prm.nchunk : prm.n_groups);
                continue;
            }
            const uint32_t uc = ua++;
            const int ab = uc % C::kABuf;
            if (!C::kATmem) {
                // the unit's A tiles (an idle stream waits too, so that its release of the
                // A buffer counts for this unit's phase)
                if (!wait(afull0 + 8u * ab, (uc / C::kABuf) & 1)) {
                    ok = false;
                    break;
                }
                if (s >= U.n_act) {
                    if (elect_one()) mbar_arrive(afree0 + 8u * ab);
                    __syncwarp();
                    it += U.n_items;
                    continue;
                }
            } else {
                if (s >= U.n_act) {
                    it += U.n_items;
                    continue;
                }
                // the unit's A tiles, copied into TMEM by the softmax warpgroup
                if (!wait(aready0 + 8u * s, ar & 1)) {
                    ok = false;
                    break;
                }
                ++ar;
            }
            tc_fence_after();
            const uint32_t a_base = smem_u32(abuf + ab * C::kABytes + s * C::kNTA * C::kATile);
            int prev_st = 0;
            for (int i = 0; i <= U.n_items; ++i) {
                const int st = it % C::kStages;
                if (i < U.n_items) {
                    if (!wait(full0 + 8u * st, (it / C::kStages) & 1)) {
                        ok = false;
                        break;
                    }
                }
                if (i > 0) {
                    // dS / P of item i - 1 written: its accumulating products
                    if (!wait(pready0 + 8u * s, pj & 1)) {
                        ok = false;
                        break;
                    }
                    ++pj;
                    if (i == 1 && nu > 0 && !wait(accfree0 + 8u * s, (nu - 1) & 1)) {
                        ok = false;
                        break;
                    }
                }
                tc_fence_after();
                if (i > 0) issue_acc(prev_st, i > 1);
                if (i < U.n_items) {
                    const uint32_t i_base = smem_u32(ring + st * C::kStage);
                    if (C::kATmem) {
                        // S = K Q^T (item tile 0); T = dY Z^T (item tile 2) + (u V) (w dZ)^T
                        // (item tile 1), with K, dY, u V in TMEM
                        const uint32_t aK = t0 + C::kColA;
#pragma unroll
                        for (int k = 0; k < D / 16; ++k) {
                            const uint64_t bd = smem_desc(i_base + 32 * k, 16, C::kSBO, C::kSwz);
                            if (elect_one()) mma_ts(t0, aK + 8 * k, bd, C::kIdescS, k > 0 ? 1u : 0u);
                            __syncwarp();
                        }
                        if (C::kLoI) {
                            // S += K lo(Q)^T (the item's last tile)
#pragma unroll
                            for (int k = 0; k < D / 16; ++k) {
                                const uint64_t bd = smem_desc(
                                    i_base + C::kNT * C::kItemTile + 32 * k, 16, C::kSBO, C::kSwz);
                                if (elect_one()) mma_ts(t0, aK + 8 * k, bd, C::kIdescS, 1u);
                                __syncwarp();
                            }
                        }
#pragma unroll
                        for (int k = 0; k < D / 16; ++k) {
                            const uint64_t bd = smem_desc(i_base + 2 * C::kItemTile + 32 * k, 16,
                                                          C::kSBO, C::kSwz);
                            if (elect_one())
                                mma_ts(t0 + C::kItem, aK + D / 2 + 8 * k, bd, C::kIdescS,
                                       k > 0 ? 1u : 0u);
                            __syncwarp();
                        }
#pragma unroll
                        for (int k = 0; k < D / 16; ++k) {
                            const uint64_t bd = smem_desc(i_base + C::kItemTile + 32 * k, 16,
                                                          C::kSBO, C::kSwz);
                            if (elect_one())
                                mma_ts(t0 + C::kItem, aK + D + 8 * k, bd, C::kIdescS, 1u);
                            __syncwarp();
                        }
                    } else {
#pragma unroll
                        for (int t = 0; t < C::kNA; ++t) {
#pragma unroll
                            for (int k = 0; k < D / 16; ++k) {
                                const uint64_t ad = smem_desc(a_base + t * C::kATile + 32 * k, 16,
                                                              C::kSBO, C::kSwz);
                                const uint64_t bd = smem_desc(i_base + t * C::kItemTile + 32 * k,
                                                              16, C::kSBO, C::kSwz);
                                if (elect_one())
                                    mma_ss(t0 + t * C::kItem, ad, bd, C::kIdescS, k > 0 ? 1u : 0u);
                                __syncwarp();
                            }
                            if (t == 0 && (C::kLoA || C::kLoI)) {
                                // S += lo(Q) K^T (the A tiles' last) or K lo(Q)^T (the item's)
                                const uint32_t a_lo = a_base + (C::kLoA ? C::kNT * C::kATile : 0);
                                const uint32_t i_lo =
                                    i_base + (C::kLoI ? C::kNT * C::kItemTile : 0);
#pragma unroll
                                for (int k = 0; k < D / 16; ++k) {
                                    const uint64_t ad =
                                        smem_desc(a_lo + 32 * k, 16, C::kSBO, C::kSwz);
                                    const uint64_t bd =
                                        smem_desc(i_lo + 32 * k, 16, C::kSBO, C::kSwz);
                                    if (elect_one()) mma_ss(t0, ad, bd, C::kIdescS, 1u);
                                    __syncwarp();
                                }
                            }
                        }
                    }
                    if (elect_one()) mma_commit(sready0 + 8u * s);
                    __syncwarp();
                    prev_st = st;
                    ++it;
                } else {
                    if (elect_one()) {
                        mma_commit(accdone0 + 8u * s);
                        if (!C::kATmem) mma_commit(afree0 + 8u * ab);
                    }
                    __syncwarp();
                    ++nu;
                }
            }
        }
        // every product issued has completed before TMEM is released
        if (elect_one()) mma_commit(fin0 + 8u * s);
        __syncwarp();
        const uint64_t tw = globaltimer_ns();
        while (!__all_sync(0xffffffffu, mbar_try_wait(fin0 + 8u * s, 0)) &&
               globaltimer_ns() - tw < prm.wait_ns) {
        }
    } else if (warp >= kFirstSoftmaxWarp && warp < kFirstSoftmaxWarp + 4 * NS) {
        // ------------------------------------------------------------ softmax warpgroups
        const int s = (warp - kFirstSoftmaxWarp) / 4;
        const int q = warp % 4;  // TMEM lane quadrant of this warp
        const int r = 32 * q + lane;
        const bool leader = q == 0 && lane == 0;
        const uint32_t t0 = tmem + ((uint32_t)(32 * q) << 16) + s * C::kColStream;
        const uint64_t c2 = pack_f32x2(prm.c, prm.c);
        uint32_t it = 0, sj = 0, na = 0, ua = 0;
        bool ok = true;
        // T23C: copy this stream's A rows of unit V (the ua-th unit of the CTA) from shared
        // memory into TMEM: K, dY, and V scaled by u = 2^(L3 - R). Every thread then releases
        // the shared-memory buffer; an idle stream only releases it.
        auto copy_a = [&](const BUnit& V, uint32_t uv) -> bool {
            const int ab = uv % C::kABuf;
            if (!warp_wait(afull0 + 8u * ab, (uv / C::kABuf) & 1, abort_flag, prm.status, prm.wait_ns))
                return false;
            if (s < V.n_act) {
                const int64_t row = V.row0 + s * kRows + r;
                const float uu =
                    row < V.rows ? exp2f(prm.Lrow[V.bh * V.rows + row] - prm.Rb[V.bh]) : 0.f;
                // the tiles are swizzled to the D-wide row (16-byte chunk k of row r at
                // k ^ (bits 7.. of the row's offset)): one-row-per-thread reads hit every bank
                const uint8_t* src = abuf + ab * C::kABytes + s * C::kNTA * C::kATile + r * D * 2;
                const int sw = ((r * D * 2) >> 7) & (D / 8 - 1);
#pragma unroll
                for (int t = 0; t < C::kNT; ++t) {
                    uint32_t v[D / 2];
                    const uint4* p4 = reinterpret_cast<const uint4*>(src + t * C::kATile);
#pragma unroll
                    for (int k = 0; k < D / 8; ++k) {
                        const uint4 x = p4[k ^ sw];
                        v[4 * k] = x.x;
                        v[4 * k + 1] = x.y;
                        v[4 * k + 2] = x.z;
                        v[4 * k + 3] = x.w;
                    }
                    if (t == 2) {
#pragma unroll
                        for (int k = 0; k < D / 2; ++k) {
                            __nv_bfloat162 b = *reinterpret_cast<__nv_bfloat162*>(&v[k]);
                            const float2 f = __bfloat1622float2(b);
                            v[k] = pack_bf16(f.x * uu, f.y * uu);
                        }
                    }
                    if (D == 16)
                        tmem_st8(t0 + C::kColA + t * (D / 2), v);
                    else
                        tmem_st16(t0 + C::kColA + t * (D / 2), v);
                }
                tmem_wait_st();
                tc_fence_before();
                mbar_arrive(aready0 + 8u * s);
            }
            mbar_arrive(afree0 + 8u * ab);
            return true;
        };
        bool copied = false;  // T23C: the current unit's A rows were copied ahead
        for (int64_t u = blockIdx.x; u < prm.n_units && ok; u += gridDim.x) {
            const BUnit U = bwd_unit<D, PASS>(prm, u);
            if (unit_skipped(prm, U.bh)) {
                u = skip_bh(U.bh, C::kRouteRows ? prm.n_groups * prm.nchunk : prm.n_groups);
                continue;
            }
            const uint32_t uc = ua++;
            if (C::kATmem) {
                if (!copied && !copy_a(U, uc)) {
                    ok = false;
                    break;
                }
                copied = false;
            }
            if (s >= U.n_act) {
                it += U.n_items;
                continue;
            }
            const int64_t row = U.row0 + s * kRows + r;
            const bool valid = row < U.rows;
            float Lr = 0.f, cr = 0.f;
            if (C::kRowStats && valid) {
                Lr = prm.Lrow[U.bh * U.rows + row];
                cr = prm.crow[U.bh * U.rows + row];
            }
            const uint64_t nLr2 = pack_f32x2(-Lr, -Lr), ncr2 = pack_f32x2(-cr, -cr);
            // T23C: u = 2^(L3 - R) of this row
            const float uu = C::kATmem && valid ? exp2f(Lr - prm.Rb[U.bh]) : 0.f;
            const uint64_t u2 = pack_f32x2(uu, uu);
            for (int i = 0; i < U.n_items; ++i, ++it) {
                const int st = it % C::kStages;
                if (!warp_wait(sready0 + 8u * s, sj & 1, abort_flag, prm.status, prm.wait_ns)) {
                    ok = false;
                    break;
                }
                ++sj;
                // S of item i complete: every product of item i - 1 is, so its stage is free
                if (i > 0 && leader) mbar_arrive(empty0 + 8u * ((it - 1) % C::kStages));
                if (C::kColStats &&
                    !warp_wait(full0 + 8u * st, (it / C::kStages) & 1, abort_flag, prm.status, prm.wait_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int nv =
                    (int)min((int64_t)C::kItem, U.item_end - (U.item0 + (int64_t)i * C::kItem));
                const float* nLc = stats + st * 2 * C::kItem;
                const float* ncc = nLc + C::kItem;
                if (nv == C::kItem)
                    bwd_item<D, PASS, true>(t0, nv, c2, nLr2, ncr2, nLc, ncc, u2);
                else
                    bwd_item<D, PASS, false>(t0, nv, c2, nLr2, ncr2, nLc, ncc, u2);
                tmem_wait_st();
                tc_fence_before();
                mbar_arrive(pready0 + 8u * s);
            }
            if (!ok) break;
            if (C::kATmem) {
                // the score products of the unit's last item are complete (its S was seen),
                // so the A rows of the CTA's next unit can go into TMEM now, ahead of this
                // unit's epilogue
                for (int64_t un = u + gridDim.x; un < prm.n_units; un += gridDim.x) {
                    const BUnit V = bwd_unit<D, PASS>(prm, un);
                    if (unit_skipped(prm, V.bh)) {
                        un = skip_bh(V.bh, prm.n_groups);
                        continue;
                    }
                    if (!copy_a(V, ua)) ok = false;
                    copied = ok;
                    break;
                }
                if (!ok) break;
            }
            // epilogue: the unit's accumulators
            if (!warp_wait(accdone0 + 8u * s, na & 1, abort_flag, prm.status, prm.wait_ns)) {
                ok = false;
                break;
            }
            ++na;
            if (leader) mbar_arrive(empty0 + 8u * ((it - 1) % C::kStages));
            tc_fence_after();
            float a0[D], a1[C::kNAcc == 2 ? D : 1];
            const uint32_t acc = t0 + C::kNA * C::kItem;
#pragma unroll
            for (int k = 0; k < D / 16; ++k) {
                uint32_t t[16];
                tmem_ld16(acc + 16 * k, t);
                tmem_wait_ld16(t);
#pragma unroll
                for (int e = 0; e < 16; ++e) a0[16 * k + e] = __uint_as_float(t[e]);
                if (C::kNAcc == 2) {
                    tmem_ld16(acc + D + 16 * k, t);
                    tmem_wait_ld16(t);
#pragma unroll
                    for (int e = 0; e < 16; ++e) a1[16 * k + e] = __uint_as_float(t[e]);
                }
            }
            tc_fence_before();
            mbar_arrive(accfree0 + 8u * s);
            if (valid) {
                if (C::kRouteRows) {
                    const int64_t idx = (U.bh * prm.nchunk + U.chunk) * prm.M + row;
                    float4* d0 = reinterpret_cast<float4*>(prm.pb + idx * D);
#pragma unroll
                    for (int k = 0; k < D / 4; ++k)
                        d0[k] = make_float4(a0[4 * k], a0[4 * k + 1], a0[4 * k + 2], a0[4 * k + 3]);
                    if (C::kNAcc == 2) {
                        float4* d1 = reinterpret_cast<float4*>(prm.pa + idx * D);
#pragma unroll
                        for (int k = 0; k < D / 4; ++k)
                            d1[k] =
                                make_float4(a1[4 * k], a1[4 * k + 1], a1[4 * k + 2], a1[4 * k + 3]);
                    }
                } else {
                    const float sc = prm.scale;
                    uint4* d0 = reinterpret_cast<uint4*>(prm.out0 + (U.bh * prm.N + row) * D);
                    uint4* d1 = reinterpret_cast<uint4*>(prm.out1 + (U.bh * prm.N + row) * D);
#pragma unroll
                    for (int k = 0; k < D / 8; ++k) {
                        uint4 v;
                        v.x = pack_bf16(sc * a0[8 * k + 0], sc * a0[8 * k + 1]);
                        v.y = pack_bf16(sc * a0[8 * k + 2], sc * a0[8 * k + 3]);
                        v.z = pack_bf16(sc * a0[8 * k + 4], sc * a0[8 * k + 5]);
                        v.w = pack_bf16(sc * a0[8 * k + 6], sc * a0[8 * k + 7]);
                        d0[k] = v;
                        v.x = pack_bf16(a1[8 * k + 0], a1[8 * k + 1]);
                        v.y = pack_bf16(a1[8 * k + 2], a1[8 * k + 3]);
                        v.z = pack_bf16(a1[8 * k + 4], a1[8 * k + 5]);
                        v.w = pack_bf16(a1[8 * k + 6], a1[8 * k + 7]);
                        d1[k] = v;
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, kTmemCols);
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

// A bf16 [z][rows][D] tensor, boxes of box_rows x D, swizzled to the row width.
bool make_map(CUtensorMap* m, const void* base, int64_t D, int64_t rows, int64_t z,
              uint32_t box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)rows, (cuuint64_t)z};
    cuuint64_t strides[2] = {(cuuint64_t)(D * 2), (cuuint64_t)(rows * D * 2)};
    cuuint32_t box[3] = {(cuuint32_t)D, box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    const CUtensorMapSwizzle sw = D == 16 ? CU_TENSOR_MAP_SWIZZLE_32B
                                          : (D == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                     : CU_TENSOR_MAP_SWIZZLE_128B);
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D, int PASS, bool LO>
cudaError_t launch_pass(const void* const* srcs, const Plan& p, BwdParams prm, cudaStream_t st) {
    using Cf = BCfg<D, PASS, LO>;
    const cudaError_t attr = ensure_smem_limit((const void*)tc_bwd_kernel<D, PASS, LO>, Cf::kSmem);
    if (attr != cudaSuccess) return attr;
    if (Cf::kRouteRows) {
        prm.n_groups = (prm.M + Cf::kGroup - 1) / Cf::kGroup;
        prm.n_units = prm.BH * prm.n_groups * prm.nchunk;
    } else {
        prm.n_groups = (prm.N + Cf::kGroup - 1) / Cf::kGroup;
        prm.n_units = prm.BH * prm.n_groups;
    }
    if (prm.n_units == 0) return cudaSuccess;
    if (Cf::kRouteRows && prm.chunk_len % Cf::kItem != 0) return cudaErrorInvalidValue;
    // A tiles: 128 rows of the pass's row dimension; items: kItem rows of the other one
    const int64_t arows = Cf::kRouteRows ? p.M : p.N;
    const int64_t irows = Cf::kRouteRows ? p.N : p.M;
    CUtensorMap maps[6];
    for (int k = 0; k < 6; ++k) {
        const bool used = (k % 3) < Cf::kNT;
        const void* base = used ? srcs[k] : srcs[k - 2];
        const bool a_side = k < 3;
        const bool per_head = a_side ? (prm.a0_per_head && k == 0) : (prm.i0_per_head && k == 3);
        if (!make_map(&maps[k], base, p.D, a_side ? arows : irows, per_head ? p.H : p.BH,
                      a_side ? (uint32_t)kRows : (uint32_t)Cf::kItem))
            return cudaErrorInvalidValue;
    }
    // Q's lo tiles (LO): an A operand of the route-row passes, an item of the token-row ones
    CUtensorMap mlo = maps[0];
    if (LO && !make_map(&mlo, srcs[6], p.D, Cf::kLoA ? arows : irows, p.BH,
                        Cf::kLoA ? (uint32_t)kRows : (uint32_t)Cf::kItem))
        return cudaErrorInvalidValue;
    int dev = 0, sms = kNumSMs;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t grid = prm.n_units < sms ? prm.n_units : sms;
    tc_bwd_kernel<D, PASS, LO><<<(unsigned)grid, Cf::kThreads, Cf::kSmem, st>>>(
        maps[0], maps[1], maps[2], maps[3], maps[4], maps[5], mlo, prm);
    return cudaGetLastError();
}

// `lo` (srcs[6] holds Q's lo operand): the hi/lo score products, for the passes whose scores
// take Q (R3, R2, T23, T23C) at D <= 32.
template <int PASS>
cudaError_t launch_d(const void* const* srcs, const Plan& p, const BwdParams& prm,
                     cudaStream_t st, bool lo) {
    constexpr bool kHasQ = PASS == kR3 || PASS == kR2 || PASS == kT23 || PASS == kT23C;
    if constexpr (kHasQ) {
        if (lo) {
            switch (p.D) {
                case 16: return launch_pass<16, PASS, true>(srcs, p, prm, st);
                case 32: return launch_pass<32, PASS, true>(srcs, p, prm, st);
                default: return cudaErrorInvalidValue;
            }
        }
    }
    if constexpr (PASS == kT23C) {
        switch (p.D) {
            case 16: return launch_pass<16, kT23C, false>(srcs, p, prm, st);
            case 32: return launch_pass<32, kT23C, false>(srcs, p, prm, st);
            default: return cudaErrorInvalidValue;
        }
    } else {
        switch (p.D) {
            case 16: return launch_pass<16, PASS, false>(srcs, p, prm, st);
            case 32: return launch_pass<32, PASS, false>(srcs, p, prm, st);
            case 64: return launch_pass<64, PASS, false>(srcs, p, prm, st);
            default: return cudaErrorInvalidValue;
        }
    }
}

}  // namespace

cudaError_t tc_bwd_pass(const Plan& p, const BwdPlan& bp, int pass, const TcBwdOperands& o,
                        float scale, int* status, cudaStream_t st) {
    const void* srcs[7] = {o.a[0], o.a[1], o.a[2], o.i[0], o.i[1], o.i[2], o.lo};
    const bool lo = o.lo != nullptr && p.D <= 32;
    BwdParams prm{};
    prm.BH = p.BH;
    prm.H = p.H;
    prm.N = p.N;
    prm.M = p.M;
    prm.c = scale * 1.4426950408889634f;
    prm.scale = scale;
    prm.a0_per_head = pass == kR1 ? 1 : 0;
    prm.i0_per_head = pass == kT1 ? 1 : 0;
    prm.chunk_len = bp.chunk_len;
    prm.nchunk = bp.nchunk;
    prm.Lrow = o.Lrow;
    prm.crow = o.crow;
    prm.Lcol = o.Lcol;
    prm.ccol = o.ccol;
    prm.pa = o.pa;
    prm.pb = o.pb;
    prm.out0 = (__nv_bfloat16*)o.out0;
    prm.out1 = (__nv_bfloat16*)o.out1;
    prm.Rb = o.Rb;
    prm.flags = o.flags;
    prm.want = o.want;
    prm.status = status;
    test_fault_for(4 + pass, &prm.wait_ns, &prm.withhold_it);
    switch (pass) {
        case kR3: return launch_d<kR3>(srcs, p, prm, st, lo);
        case kR2: return launch_d<kR2>(srcs, p, prm, st, lo);
        case kR1: return launch_d<kR1>(srcs, p, prm, st, false);
        case kT23: return launch_d<kT23>(srcs, p, prm, st, lo);
        case kT1: return launch_d<kT1>(srcs, p, prm, st, false);
        case kT23C: return launch_d<kT23C>(srcs, p, prm, st, lo);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace flarepp
