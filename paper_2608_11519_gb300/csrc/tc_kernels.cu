// Tensor-core (tcgen05 / TMEM / TMA) kernels of the routing chain: the bf16 dtype path.
//
// One warp-specialised kernel template serves both directions of the routing chain
// (Sec. 3.2, eqs. flarepp_dynamic_query and flarepp_mixer):
//
//   encode (calls 1, 2): TMEM lanes are routes. A group of NS route tiles (128 routes
//     each; the A operand: seeds or Q) meets a stream of items of kItem tokens (K and V
//     tiles) from one chunk of the sequence. Each route row keeps an online softmax over
//     tokens, and the CTA writes per-chunk partials (reference, sum, unnormalised value sum)
//     for the log-sum-exp merge of App. A.3.
//   decode (call 3): TMEM lanes are tokens. A group of NS token tiles (K, 128 tokens each)
//     meets a stream of items of kItem routes (Q and Z tiles). Each token row keeps an
//     online softmax over routes and writes its normalised row of Y.
//
// Work is cut into four TMEM "streams". Stream s owns one score buffer of 128 x kItem fp32
// (S is rewritten in place as bf16 P, the A operand of the PV product) and a 128 x D fp32
// accumulator O (two in the decode at D <= 32, one per unit parity), and reads one resident A
// tile in shared memory, so that S = A * B^T is a SMEM x SMEM product and all TMEM columns go
// to S and O. The decode double-buffers its A tiles, so the next unit's tiles land while the
// current unit runs. Roles (24 warps, a register split gives warpgroups 0 and 1 40 registers
// per thread and the four softmax warpgroups 96):
//   warps 0..3    one MMA warp per stream: for item j, the PV of item j-1 and the S of
//                 item j, then one commit, all issued from one elected lane (a commit
//                 stalls only the warp that issues it)
//   warp 4        the TMA producer (A tiles and the item ring, K/V or Q/Z, all swizzled to
//                 one D-wide row), with blocking waits; warps 5..7 only take part in the split
//   warps 8..23   four softmax warpgroups; warpgroup s serves stream s (four warps per SMSP
//                 hide each other's latencies)
// Each launch is a pair of kernels on the stream. The fast kernel keeps, per row, the first
// score of the unit as its reference m (any score of the row is a valid reference: it alone
// adds 2^0 to the sum) and computes P = 2^(c S - m) with no maximum pass, storing P chunk by
// chunk. An item whose probabilities sum past 2^48 (a score far above the reference) cannot
// be repaired there: the kernel raises the launch's overflow word when it ends, and the safe
// kernel after it, which otherwise returns at once, recomputes the launch with the exact
// maximum wherever the sum passes that limit.
// Every wait is bounded (2 s of %globaltimer, or the test hook's limit): on expiry the
// kernel records FLAREPP_ERR_TIMEOUT in the status word, every role leaves its loops, the
// producer waits for its copies in flight, and TMEM is freed.
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

constexpr int kWarps = 24;
constexpr int kThreads = kWarps * 32;
constexpr int kProducerWarp = 4;      // warpgroup 1: the TMA producer and three idle warps
constexpr int kFirstSoftmaxWarp = 8;
// Registers per thread after the split (launch: 80 x 768 threads): warpgroups 0 (MMA) and 1
// (producer) lower to 40, the four softmax warpgroups raise to 96.
constexpr uint32_t kRegsControl = 40;
constexpr uint32_t kRegsSoftmax = 96;
static_assert(kRegsControl * 256 + kRegsSoftmax * 512 <= 80 * 768, "register split");
constexpr int NS = 4;           // TMEM streams
constexpr int kTileRows = 128;  // TMEM lanes, MMA M
constexpr uint64_t kDefaultWaitNs = 2000000000ull;
constexpr uint32_t kTmemCols = 512;
constexpr float kLog2e = 1.4426950408889634f;
// Sum of one item's probabilities above which the reference max is recomputed exactly.
constexpr float kFastLimit = 281474976710656.0f;  // 2^48

// LO (the training forward, D <= 32): Q enters the scores of calls 2 and 3 as a pair of bf16
// operands, hi = bf16(Q) and lo = bf16(Q - hi), and each score product is the sum of the two
// products (S = (hi + lo) B^T in the encode of call 2, S = A (hi + lo)^T in the decode), so the
// scores see Q to about 2^-17 instead of bf16's 2^-9. The encode keeps both A tiles in its
// shared-memory A buffer (the lo tile after the hi tile); the decode's items carry Q's lo tile
// as a third tile.
template <int D, bool DEC, bool LO = false>
struct Cfg {
    static_assert(!LO || D <= 32, "the hi/lo form of Q serves D = 16 and 32");
    static constexpr bool kLoA = LO && !DEC;  // encode of call 2: A = Q as hi and lo tiles
    static constexpr bool kLoB = LO && DEC;   // decode: every item also carries Q's lo tile
    static constexpr int kANum = kLoA ? 2 : 1;  // A tiles per stream
    // The A tiles (the route tiles in the encode, the token tiles in the decode) stay in shared
    // memory where the TMA puts them, swizzled like the ring tiles, and the MMAs read them there
    // (`ss` score products); nothing copies them into TMEM, so all 512 columns go to the score
    // tiles and accumulators. The encode's units are long (hundreds of items): one A buffer,
    // and items of 96 tokens (112 at D = 16; 64 at D = 64: S 4 x 64 + O 4 x 64 columns), so
    // the per-item round trip is paid once per 96 tokens. The decode's units are only M/64
    // items, so per-unit costs show: its A tiles are double-buffered so the next unit's land
    // during this one, and where TMEM has the room (D <= 32) it keeps two O accumulators per
    // stream, one per unit parity, so that a unit's epilogue can wait until the next unit's
    // first item is under way; at D = 64 the columns instead widen its items to 48 routes
    // (S 4 x 48 + O 4 x 64).
    static constexpr int kItem = D == 64 ? (DEC ? 48 : 64) : (DEC ? 64 : (D == 16 ? 112 : 96));
    static constexpr int B = 1;                         // score buffers per stream
    // shared-memory A buffers (four for the decode at small M measured no faster than two)
    static constexpr int kABufS = DEC ? 2 : 1;
    static constexpr int kAAhead = kABufS > 1 ? kABufS - 1 : 1;  // units the A copies run ahead
    static constexpr int kOBuf = (DEC && D <= 32) ? 2 : 1;    // O accumulators per stream
    static constexpr int kGroup = NS * kTileRows;     // resident rows per work unit
    static constexpr int kATile = kTileRows * D * 2;  // one 128-row operand tile
    static constexpr int kABytes = NS * kANum * kATile;
    static constexpr int kItemTile = kItem * D * 2;
    static constexpr int kStage = (kLoB ? 3 : 2) * kItemTile;
    static constexpr uint32_t kSwz = D == 16 ? kSw32 : (D == 32 ? kSw64 : kSw128);
    static constexpr uint32_t kSBO = 8 * D * 2;  // bytes between 8-row groups
    // Ring items. A stream that takes every n_par-th item (an encode unit with fewer than four
    // route tiles gives each stream one token parity) looks ahead only kStages / n_par of its
    // own items, and the copy of its next item cannot start before the stream frees the stage
    // kStages items back; so the encode takes as many stages as shared memory holds, up to 16.
    // The decode's streams take every item, and 8 stages cover the copy latency.
    static constexpr int kStagesFit = (232448 - 2048 - kABufS * kABytes) / kStage;
    static constexpr int kStages = DEC ? 8 : (kStagesFit < 16 ? kStagesFit : 16);
    // barriers: full[S], empty[S], a_full[kABufS] (a unit's A tiles landed), a_free[kABufS]
    //           (one arrive per softmax warpgroup once it has seen the unit's last S: the
    //           buffer may be refilled), sync[NS][2] = {s_ready, o_done} per stream (S of an
    //           item complete; every PV of the stream's unit complete), p_ready[NS][2] (slot 0
    //           used). With two O accumulators a decode unit's last PV goes out with the next
    //           unit's first S, so o_done is committed only for a CTA's last unit. A barrier that
    //           a warp waits on by parity never runs two phases ahead of that warp: s_ready of
    //           the next item needs this item's P (p_ready counts every warp of the warpgroup),
    //           o_done of the next unit needs that unit's P, a_full of unit k + kABufS needs
    //           a_free of unit k.
    static constexpr int kNumBars = 2 * kStages + 2 * kABufS + 4 * NS;
    static constexpr int kData = kABufS * kABytes + kStages * kStage;
    static constexpr int kNeed = 1024 + kData + kNumBars * 8 + 16;
    // at least 120 KB so that one CTA owns an SM and its 512 TMEM columns
    static constexpr int kSmem = kNeed > 122880 ? kNeed : 122880;
    static constexpr uint32_t kIdescS = idesc_bf16_f32(128, kItem, false, false);
    static constexpr uint32_t kIdescPV = idesc_bf16_f32(128, D, false, true);
    // TMEM columns
    static constexpr uint32_t kColS = 0;               // NS x B x kItem
    static constexpr uint32_t kColO = NS * B * kItem;  // kOBuf x NS x D
    static_assert(kColO + kOBuf * NS * D <= kTmemCols, "TMEM budget");
    static_assert(kSmem <= 232448, "shared memory budget");
    static_assert(kStages >= 2 * B * NS, "ring depth: the full wait precedes the PV");
    static_assert(B == 1, "the s_ready / o_done protocol has one score buffer per stream");
};

struct TcParams {
    int64_t BH, H, N, M;
    int a_per_head;  // encode call 1: the A operand (seeds) is indexed by head
    float c;         // |scale| * log2(e)
    int64_t chunk_len, nchunk, n_groups;
    float* pmax;
    float* psum;
    float* pacc;
    int64_t n_tok_groups;
    __nv_bfloat16* Y;
    float* lse;  // decode: each token's base-2 log-normaliser, or null
    int64_t n_units;
    int* status;
    int* overflow;  // raised by the fast kernel; the safe kernel runs only when it is set
    uint64_t wait_ns;     // bound of every wait (kDefaultWaitNs unless the test hook is set)
    int64_t withhold_it;  // test hook: ring item of CTA 0 the producer never loads (-1: none)
};

// route tiles of encode group g, rounded up to 1, 2 or 4 (a divisor of the stream count)
__device__ __forceinline__ int na_of_group(int64_t M, int64_t g) {
    const int64_t rem = M - g * NS * kTileRows;
    const int64_t tiles = rem >= NS * kTileRows ? NS : (rem + kTileRows - 1) / kTileRows;
    return tiles <= 1 ? 1 : (tiles <= 2 ? 2 : 4);
}

struct Unit {
    int64_t bh, chunk, g, tg;
    int zA, rowA0, zB;
    int n_a, n_par, n_items;
    int64_t item0, item_end;
};

// The plan keeps unit counts, and so every quotient below, within 32 bits; 32-bit divisions by
// runtime values cost a few instructions where 64-bit ones cost about seventy.
template <int D, bool DEC, bool LO>
__device__ __forceinline__ Unit get_unit(const TcParams& p, int64_t u64) {
    using C = Cfg<D, DEC, LO>;
    const uint32_t u = (uint32_t)u64;
    Unit U;
    if (DEC) {
        const uint32_t ntg = (uint32_t)p.n_tok_groups;
        U.tg = u % ntg;
        U.bh = u / ntg;
        U.chunk = 0;
        U.g = 0;
        U.zA = (int)U.bh;
        U.rowA0 = (int)(U.tg * C::kGroup);
        U.n_a = NS;
        U.n_par = 1;
        U.item0 = 0;
        U.item_end = p.M;
    } else {
        const uint32_t nchunk = (uint32_t)p.nchunk, ngroups = (uint32_t)p.n_groups;
        U.chunk = u % nchunk;
        const uint32_t t = u / nchunk;
        U.g = t % ngroups;
        U.bh = t / ngroups;
        U.tg = 0;
        U.zA = (int)(p.a_per_head ? (uint32_t)U.bh % (uint32_t)p.H : (uint32_t)U.bh);
        U.rowA0 = (int)(U.g * C::kGroup);
        U.n_a = na_of_group(p.M, U.g);
        U.n_par = NS / U.n_a;
        U.item0 = U.chunk * p.chunk_len;
        U.item_end = min(p.N, U.item0 + p.chunk_len);
    }
    U.zB = (int)U.bh;
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
// The same wait taken by a whole warp: true only if every lane saw the phase complete.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          int* status, uint64_t limit) {
    const bool got = wait_bar(bar, parity, abort_flag, status, limit);
    return __all_sync(0xffffffffu, got);
}

// ------------------------------------------------------------------ softmax helpers

// Online-softmax state of one TMEM stream, held by every thread of its warpgroup for its row.
struct SoftmaxStream {
    int s;          // stream index
    int par;        // token parity of the stream's items in this unit (s / n_a)
    int cnt, j;     // items of the stream in this unit, items done
    int ob;         // O accumulator of this unit (0, or the unit's parity with two)
    int ab;         // shared-memory A buffer of this unit
    float m, l;     // reference max (base 2, scaled) and running sum
    uint32_t ph0;   // s_ready phases completed in earlier units (one per item)
    uint32_t od;    // o_done phases consumed (one per unit whose end waits on it)
    bool over;      // fast kernel: some item's sum passed kFastLimit
    __device__ __forceinline__ void begin(const Unit& U) {
        par = s / U.n_a;
        cnt = U.n_items > par ? (U.n_items - par + U.n_par - 1) / U.n_par : 0;
        j = 0;
        m = -INFINITY;
        l = 0.f;
    }
};

// Max over the valid columns [0, nv) of one chunk of W = 32 or 16 columns (columns
// base .. base + W - 1).
template <int W>
__device__ __forceinline__ float chunk_max(const uint32_t* sr, int base, int nv) {
    float a0 = -INFINITY, a1 = -INFINITY, a2 = -INFINITY, a3 = -INFINITY;
    if (base + W <= nv) {
#pragma unroll
        for (int k = 0; k < W; k += 8) {
            a0 = max3f(a0, __uint_as_float(sr[k]), __uint_as_float(sr[k + 1]));
            a1 = max3f(a1, __uint_as_float(sr[k + 2]), __uint_as_float(sr[k + 3]));
            a2 = max3f(a2, __uint_as_float(sr[k + 4]), __uint_as_float(sr[k + 5]));
            a3 = max3f(a3, __uint_as_float(sr[k + 6]), __uint_as_float(sr[k + 7]));
        }
    } else {
#pragma unroll
        for (int k = 0; k < W; ++k)
            if (base + k < nv) a0 = fmaxf(a0, __uint_as_float(sr[k]));
    }
    return max3f(a0, a1, fmaxf(a2, a3));
}

// P = 2^(c S - m) for one chunk of W = 32 or 16 columns, packed bf16 pairs into
// pr[0 .. W/2); returns the chunk's row sum. Columns at or beyond nv are not part of the
// softmax: probability 0.
template <int W>
__device__ __forceinline__ float exp_chunk(const uint32_t* sr, uint32_t* pr, int base, int nv,
                                           float c, uint64_t c2, float m) {
    if (base + W <= nv) {
        const uint64_t nm2 = pack_f32x2(-m, -m);
        uint64_t acc0 = 0, acc1 = 0;  // two packed (lo, hi) partial sums
#pragma unroll
        for (int k = 0; k < W / 2; k += 2) {
            pr[k] = exp2_pair(__uint_as_float(sr[2 * k]), __uint_as_float(sr[2 * k + 1]), c2,
                              nm2, acc0);
            pr[k + 1] = exp2_pair(__uint_as_float(sr[2 * k + 2]), __uint_as_float(sr[2 * k + 3]),
                                  c2, nm2, acc1);
        }
        float a, b, x, y;
        unpack_f32x2(acc0, a, b);
        unpack_f32x2(acc1, x, y);
        return (a + b) + (x + y);
    }
    float t0 = 0.f, t1 = 0.f;
#pragma unroll
    for (int k = 0; k < W / 2; ++k) {
        const float p0 =
            base + 2 * k < nv ? ex2(fmaf(__uint_as_float(sr[2 * k]), c, -m)) : 0.f;
        const float p1 =
            base + 2 * k + 1 < nv ? ex2(fmaf(__uint_as_float(sr[2 * k + 1]), c, -m)) : 0.f;
        t0 += p0;
        t1 += p1;
        pr[k] = pack_bf16(p0, p1);
    }
    return t0 + t1;
}

// P for a whole item tile of ITEM columns at TMEM column scol (S is read 32 columns at a
// time, and a last 16 when ITEM is an odd multiple of 16); packed bf16 pairs go to
// pr[0 .. ITEM/2). Returns the
// row sum. With FIRST_REF and
// `first` the reference m is first set to the row's own first score, c S[0]: any score of
// the row is a valid reference (that score alone contributes 2^0 = 1 to the sum, so the
// sum never underflows), and a reference far below the row's maximum shows up as a sum
// past the fast-path limit, which sends the item to the exact-max path.
//
// STORE (the fast kernel): each chunk's P goes back to TMEM as soon as it is packed (it covers
// only columns already read), so S is gone by the end. Otherwise P stays in pr for the
// caller, and S stays intact until the caller writes it.
template <int ITEM, bool FIRST_REF, bool STORE>
__device__ __forceinline__ float exp_tile(uint32_t scol, uint32_t* pr, int nv, float c,
                                          uint64_t c2, float& m, bool first) {
    float sum = 0.f;
#pragma unroll
    for (int h = 0; h < ITEM / 32; ++h) {
        uint32_t sr[32];
        tmem_ld32(scol + 32 * h, sr);
        tmem_wait_ld32(sr);
        if (FIRST_REF && h == 0 && first) m = c * __uint_as_float(sr[0]);
        sum += exp_chunk<32>(sr, pr + 16 * h, 32 * h, nv, c, c2, m);
        if constexpr (STORE) tmem_st16(scol + 16 * h, pr + 16 * h);
    }
    if constexpr (ITEM % 32 == 16) {
        constexpr int base = ITEM - 16;
        uint32_t sr[16];
        tmem_ld16(scol + base, sr);
        tmem_wait_ld16(sr);
        sum += exp_chunk<16>(sr, pr + base / 2, base, nv, c, c2, m);
        if constexpr (STORE) tmem_st8(scol + base / 2, pr + base / 2);
    }
    return sum;
}

// P of a whole item (ITEM / 2 packed words) to TMEM column scol, 32, 16 and 8 words at a time.
template <int ITEM>
__device__ __forceinline__ void store_p(uint32_t scol, uint32_t* pr) {
    constexpr int W = ITEM / 2;
    static_assert(W % 8 == 0, "P comes in multiples of 8 words");
#pragma unroll
    for (int w = 0; w + 32 <= W; w += 32) tmem_st32(scol + w, pr + w);
    constexpr int w16 = W / 32 * 32;
    if constexpr (W - w16 >= 16) tmem_st16(scol + w16, pr + w16);
    constexpr int w8 = w16 + (W - w16 >= 16 ? 16 : 0);
    if constexpr (W - w8 >= 8) tmem_st8(scol + w8, pr + w8);
}

// One item of this warpgroup's stream for this thread's row: read S, update the online
// softmax, write P back over S, signal the stream's MMA warp. S of item j being ready
// means the PV of item j - B has completed, so the warpgroup leader frees that item's ring
// stage; the S of the unit's last item was the last product to read the unit's A tiles, so
// the leader then also frees the A buffer. Returns false when the kernel is aborting.
//   fast kernel (!SAFE): the reference is kept from the items before (a unit's first item
//     takes its first score) and P is stored chunk by chunk, so S is gone by the end of the
//     item. A sum past kFastLimit (a score far above the reference) cannot be repaired
//     here: the thread notes it, the kernel raises the launch's overflow word when it ends,
//     and the safe kernel that follows on the stream recomputes the whole launch.
//   safe kernel: P is stored once the item's sum is known; a sum past kFastLimit sends the
//     item to the exact-max path, which reads S again (the decode, whose units are short,
//     takes the first item's reference from its first score; the encode, whose units are
//     long, takes the first item's exact maximum).
template <int D, bool DEC, bool SAFE, bool LO>
__device__ __forceinline__ bool softmax_step(SoftmaxStream& S, const Unit& U, uint32_t tmem,
                                             uint32_t lane_off, float c, uint64_t c2,
                                             uint32_t sready_s, uint32_t pready_s, uint32_t empty0,
                                             uint32_t afree0, bool wg_leader, uint32_t it0,
                                             volatile int* abort_flag, int* status,
                                             uint64_t limit, volatile int* overflow) {
    using C = Cfg<D, DEC, LO>;
    const int j = S.j;
    const int b = j % C::B;
    const uint32_t par_j = (S.ph0 + (uint32_t)j) & 1u;
    if (!warp_wait(sready_s + 8u * b, par_j, abort_flag, status, limit)) return false;
    tc_fence_after();
    const int par = S.par;
    if (wg_leader && j >= C::B) {
        const int i_old = par + (j - C::B) * U.n_par;
        mbar_arrive(empty0 + 8u * ((it0 + i_old) % C::kStages));
    }
    // the unit's last S is complete, so its MMAs no longer read the A buffer. Stream 0 (which
    // always has items) also arrives for the streams with no item in the unit (short encode
    // chunks split by token parity), which do not arrive themselves: arriving at once, such a
    // stream could arrive for the next unit as well before a slower stream arrived for this
    // one, completing this unit's phase of a_free while that stream's last S still reads.
    if (wg_leader && j == S.cnt - 1) {
        uint32_t n = 1;
        if constexpr (!DEC)
            if (S.s == 0 && U.n_items < U.n_par) n += U.n_a * (U.n_par - U.n_items);
        mbar_arrive_n(afree0 + 8u * S.ab, n);
    }
    const int item = par + j * U.n_par;
    const int64_t start = U.item0 + (int64_t)item * C::kItem;
    const int nv = (int)min((int64_t)C::kItem, U.item_end - start);
    const uint32_t scol = tmem + lane_off + C::kColS + (S.s * C::B + b) * C::kItem;
    uint32_t pr[C::kItem / 2];
    float sum = 0.f;
    if constexpr (!SAFE) {
        sum = exp_tile<C::kItem, true, true>(scol, pr, nv, c, c2, S.m, j == 0);
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(pready_s + 8u * b);
        S.over |= !(sum <= kFastLimit);  // checked once, when the kernel ends
        S.l += sum;
        ++S.j;
        return true;
    }
    bool slow = !DEC && j == 0;
    if (!slow) {
        sum = exp_tile<C::kItem, DEC, false>(scol, pr, nv, c, c2, S.m, j == 0);
        slow = __any_sync(0xffffffffu, !(sum <= kFastLimit));
    }
    if (slow) {
        // exact max of this item (S is still intact in TMEM: P has not been written yet)
        float mx = -INFINITY;
#pragma unroll
        for (int h = 0; h < C::kItem / 32; ++h) {
            uint32_t sr[32];
            tmem_ld32(scol + 32 * h, sr);
            tmem_wait_ld32(sr);
            mx = fmaxf(mx, chunk_max<32>(sr, 32 * h, nv));
        }
        if (C::kItem % 32 == 16) {
            uint32_t sr[16];
            tmem_ld16(scol + C::kItem - 16, sr);
            tmem_wait_ld16(sr);
            mx = fmaxf(mx, chunk_max<16>(sr, C::kItem - 16, nv));
        }
        const float cand = mx * c;
        bool need = false;
        float alpha = 1.f;
        if (cand > S.m) {
            alpha = ex2(S.m - cand);  // 0 when S.m is -inf
            need = j > 0;
            S.l *= alpha;
            S.m = cand;
        }
        if (__any_sync(0xffffffffu, need)) {
            // (the PV of item j - 1 is complete: S of item j followed it in the tensor pipe)
            const uint32_t ocol = tmem + lane_off + C::kColO + (S.ob * NS + S.s) * D;
            const float f = need ? alpha : 1.f;
#pragma unroll
            for (int k = 0; k < D / 16; ++k) {
                uint32_t o[16];
                tmem_ld16(ocol + 16 * k, o);
                tmem_wait_ld16(o);
#pragma unroll
                for (int e = 0; e < 16; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * f);
                tmem_st16(ocol + 16 * k, o);
            }
        }
        sum = exp_tile<C::kItem, false, false>(scol, pr, nv, c, c2, S.m, false);
    }
    S.l += sum;
    store_p<C::kItem>(scol, pr);
    tmem_wait_st();
    tc_fence_before();
    mbar_arrive(pready_s + 8u * b);
    ++S.j;
    return true;
}

// The end of one unit of the stream, for this row: the unit's online-softmax state (m, l),
// its item count, the ring item its items start from, its O accumulator and (decode) its A
// buffer. Wait until all of the unit's PVs are complete, free the ring stage of the last item
// (and, if the stream had no items, the unit's shared-memory A buffer), read O and write the
// unit's result (the chunk partial in the encode, the normalised output row of Y in the
// decode).
// `deferred`: the decode with two O accumulators runs this one unit late, after the next
// unit's first item, whose s_ready was committed after the unit's last PV (the MMA warp
// issues the two together); otherwise the wait is on o_done.
struct UnitEnd {
    float m, l;
    int cnt, ob, ab;
    uint32_t it0;
};

template <int D, bool DEC, bool LO>
__device__ __forceinline__ bool finish_stream(SoftmaxStream& S, const UnitEnd& E, const Unit& U,
                                              const TcParams& prm, uint32_t tmem,
                                              uint32_t lane_off, int r, uint32_t sready_s,
                                              uint32_t empty0, uint32_t afree0, bool wg_leader,
                                              bool deferred, volatile int* abort_flag) {
    using C = Cfg<D, DEC, LO>;
    const int a = S.s % U.n_a;
    const int par = S.s / U.n_a;
    float o[D];
    if (E.cnt > 0) {
        if (!deferred) {
            if (!warp_wait(sready_s + 8u, S.od & 1u, abort_flag, prm.status, prm.wait_ns))
                return false;
            ++S.od;
            tc_fence_after();
        }
        if (wg_leader) {
            for (int jj = E.cnt - C::B < 0 ? 0 : E.cnt - C::B; jj < E.cnt; ++jj) {
                const int i_old = par + jj * U.n_par;
                mbar_arrive(empty0 + 8u * ((E.it0 + i_old) % C::kStages));
            }
        }
        const uint32_t ocol = tmem + lane_off + C::kColO + (E.ob * NS + S.s) * D;
        // every load of O in flight before one wait
        uint32_t t[D];
        if (D == 16) {
            tmem_ld16(ocol, t);
            tmem_wait_ld16(t);
        } else {
#pragma unroll
            for (int kk = 0; kk < D / 32; ++kk) tmem_ld32(ocol + 32 * kk, t + 32 * kk);
#pragma unroll
            for (int kk = 0; kk < D / 32; ++kk) tmem_wait_ld32(t + 32 * kk);
        }
#pragma unroll
        for (int d = 0; d < D; ++d) o[d] = __uint_as_float(t[d]);
    } else {
#pragma unroll
        for (int d = 0; d < D; ++d) o[d] = 0.f;
    }
    if (DEC) {
        const int64_t tok = U.tg * C::kGroup + a * kTileRows + r;
        if (tok < prm.N) {
            const float inv = 1.f / E.l;
            uint4* dst = reinterpret_cast<uint4*>(prm.Y + (U.bh * prm.N + tok) * D);
#pragma unroll
            for (int kk = 0; kk < D / 8; ++kk) {
                uint4 v;
                v.x = pack_bf16(o[8 * kk + 0] * inv, o[8 * kk + 1] * inv);
                v.y = pack_bf16(o[8 * kk + 2] * inv, o[8 * kk + 3] * inv);
                v.z = pack_bf16(o[8 * kk + 4] * inv, o[8 * kk + 5] * inv);
                v.w = pack_bf16(o[8 * kk + 6] * inv, o[8 * kk + 7] * inv);
                dst[kk] = v;
            }
            if (prm.lse) prm.lse[U.bh * prm.N + tok] = E.m + log2f(E.l);
        }
    } else {
        const int64_t route = U.g * C::kGroup + a * kTileRows + r;
        if (route < prm.M) {
            const int64_t idx = (U.bh * (prm.nchunk * 4) + U.chunk * 4 + par) * prm.M + route;
            prm.pmax[idx] = E.cnt > 0 ? E.m : -INFINITY;
            prm.psum[idx] = E.l;
            float4* dst = reinterpret_cast<float4*>(prm.pacc + idx * D);
#pragma unroll
            for (int kk = 0; kk < D / 4; ++kk)
                dst[kk] = make_float4(o[4 * kk], o[4 * kk + 1], o[4 * kk + 2], o[4 * kk + 3]);
        }
    }
    return true;
}

// ------------------------------------------------------------------ the kernel

template <int D, bool DEC, bool SAFE, bool LO>
__global__ void __launch_bounds__(kThreads, 1)
    tc_chain_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmL,
                    const TcParams prm) {
    using C = Cfg<D, DEC, LO>;
    pdl_trigger();
    if constexpr (SAFE) {
        // the safe kernel recomputes the launch only when the fast one overflowed
        __shared__ int run;
        pdl_wait();
        if (threadIdx.x == 0) run = *reinterpret_cast<volatile int*>(prm.overflow);
        __syncthreads();
        if (!run) return;
    }
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    uint8_t* abuf = smem;                         // kABufS x NS x kANum A tiles
    // kStages x (B tile, C tile[, lo tile]), swizzled like the A tiles
    uint8_t* ring = smem + C::kABufS * C::kABytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(ring + C::kStages * C::kStage);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::kNumBars);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const uint32_t full0 = smem_u32(bars);
    const uint32_t empty0 = full0 + 8u * C::kStages;
    const uint32_t afull0 = full0 + 8u * (2 * C::kStages);
    const uint32_t afree0 = afull0 + 8u * C::kABufS;
    const uint32_t sready0 = afree0 + 8u * C::kABufS;  // [NS][2]
    const uint32_t pready0 = sready0 + 16u * NS;  // [NS][2]

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int st = 0; st < C::kStages; ++st) {
            mbar_init(full0 + 8u * st, 1);
            mbar_init(empty0 + 8u * st, NS);
        }
        for (int b = 0; b < C::kABufS; ++b) {
            mbar_init(afull0 + 8u * b, 1);
            mbar_init(afree0 + 8u * b, NS);
        }
        for (int s = 0; s < NS; ++s) {
            mbar_init(sready0 + 16u * s, 1);
            mbar_init(sready0 + 16u * s + 8u, 1);
            mbar_init(pready0 + 16u * s, 128);
            mbar_init(pready0 + 16u * s + 8u, 128);
        }
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmA);
        prefetch_tmap(&tmB);
        prefetch_tmap(&tmC);
        if constexpr (LO) prefetch_tmap(&tmL);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // every global access below may depend on the kernel before this one
    pdl_wait();

    if (warp < kProducerWarp) {
        // ------------------------------------------------------------ MMA warps
        // Warp s drives stream s. For each of its items: the PV of its previous item (P
        // from TMEM, V or Z from the ring), the S of this item (A from TMEM in the encode, from
        // shared memory in the decode; K or Q from the ring) and one commit, which the softmax
        // waits on, all from one elected lane with descriptors derived from precomputed ones.
        // It observes the full barrier of every ring item in order, so each parity test names
        // one phase.
        regs_lower<kRegsControl>();
        const int s = warp;
        const uint32_t ring_u = smem_u32(ring);
        const uint64_t dS0 = smem_desc(ring_u, 16, C::kSBO, C::kSwz);
        const uint64_t dV0 = smem_desc(ring_u + C::kItemTile, C::kItemTile, C::kSBO, C::kSwz);
        const uint64_t dA0 = smem_desc(smem_u32(abuf), 16, C::kSBO, C::kSwz);
        const uint32_t d_s = tmem + C::kColS + s * C::kItem;  // B = 1: one score buffer
        const uint32_t sready_s = sready0 + 16u * s;
        const uint32_t pready_s = pready0 + 16u * s;
        uint32_t it = 0, ua = 0, pc = 0;  // ring items seen, units, p_ready phases consumed
        // The PV owed for the stream's previous item (its ring stage, the O accumulator it adds
        // into, whether it adds or starts it) goes out with the next S under one commit. In the
        // decode with two O accumulators it crosses unit boundaries too: a unit then ends with
        // no commit of its own, and s_ready of the next unit's first item also says that the
        // unit's O is final and its A tile no longer read.
        bool pv_owed = false;
        uint32_t pv_st = 0, pv_o = 0, pv_acc = 0;
        bool ok = true;
        for (int64_t u = blockIdx.x; u < prm.n_units && ok; u += gridDim.x, ++ua) {
            const Unit U = get_unit<D, DEC, LO>(prm, u);
            const int a = s % U.n_a;
            const int par = s / U.n_a;
            // the unit's A tile: shared-memory buffer ua % kABufS as the TMA wrote it
            const int ab = ua % C::kABufS;
            if (!warp_wait(afull0 + 8u * ab, (ua / C::kABufS) & 1, abort_flag, prm.status,
                           prm.wait_ns))
                break;
            const uint64_t dA = dA0 + ((uint64_t)(ab * C::kABytes + a * C::kANum * C::kATile) >> 4);
            // O accumulator of this unit: the unit's parity with two, else the only one (the A
            // buffer index above runs to kABufS - 1 and must not pick it)
            const int ob = C::kOBuf == 2 ? (int)(ua & 1) : 0;
            const uint32_t d_o = tmem + C::kColO + (ob * NS + s) * D;
            int j = 0;
            for (int i = 0; i < U.n_items; ++i, ++it) {
                const uint32_t st = it % C::kStages;
                // the item's full barrier first (the softmax is still busy with item j - 1, so
                // this wait is off the P -> PV -> S round trip), then the P of item j - 1.
                // Item i lands once item i - kStages is released; with kStages >= 2 NS that
                // item's PV was issued in an earlier iteration, so this wait closes no cycle.
                if (!warp_wait(full0 + 8u * st, (it / C::kStages) & 1, abort_flag, prm.status, prm.wait_ns)) {
                    ok = false;
                    break;
                }
                if ((i & (U.n_par - 1)) != par) continue;
                if (pv_owed) {
                    if (!warp_wait(pready_s, pc & 1, abort_flag, prm.status, prm.wait_ns)) {
                        ok = false;
                        break;
                    }
                    ++pc;
                }
                tc_fence_after();
                if (elect_one()) {
                    if (pv_owed) {
                        const uint64_t dv = dV0 + ((pv_st * C::kStage) >> 4);
#pragma unroll
                        for (int k = 0; k < C::kItem / 16; ++k)
                            mma_ts(pv_o, d_s + 8 * k, dv + (uint64_t)(2 * D * k), C::kIdescPV,
                                   (pv_acc || k > 0) ? 1u : 0u);
                    }
                    const uint64_t ds = dS0 + ((st * C::kStage) >> 4);
#pragma unroll
                    for (int k = 0; k < D / 16; ++k)
                        mma_ss(d_s, dA + (uint64_t)(2 * k), ds + (uint64_t)(2 * k), C::kIdescS,
                               k > 0 ? 1u : 0u);
                    if constexpr (C::kLoA) {
                        // S += lo(Q) K^T: the lo tile follows the hi tile
                        const uint64_t dAl = dA + (uint64_t)(C::kATile >> 4);
#pragma unroll
                        for (int k = 0; k < D / 16; ++k)
                            mma_ss(d_s, dAl + (uint64_t)(2 * k), ds + (uint64_t)(2 * k), C::kIdescS,
                                   1u);
                    }
                    if constexpr (C::kLoB) {
                        // S += K lo(Q)^T: the item's third tile
                        const uint64_t dl = ds + (uint64_t)((2 * C::kItemTile) >> 4);
#pragma unroll
                        for (int k = 0; k < D / 16; ++k)
                            mma_ss(d_s, dA + (uint64_t)(2 * k), dl + (uint64_t)(2 * k), C::kIdescS,
                                   1u);
                    }
                    mma_commit(sready_s);
                }
                __syncwarp();
                pv_owed = true;
                pv_st = st;
                pv_o = d_o;
                pv_acc = j > 0 ? 1u : 0u;
                ++j;
            }
            if (!ok) break;
            // decode with two O accumulators: the last PV goes out with the next unit's first S
            if (C::kOBuf == 2 && u + gridDim.x < prm.n_units) continue;
            // the PV of the unit's last item, then o_done: O is final for the softmax
            if (pv_owed && !warp_wait(pready_s, pc & 1, abort_flag, prm.status, prm.wait_ns)) break;
            if (pv_owed) ++pc;
            tc_fence_after();
            if (elect_one()) {
                if (pv_owed) {
                    const uint64_t dv = dV0 + ((pv_st * C::kStage) >> 4);
#pragma unroll
                    for (int k = 0; k < C::kItem / 16; ++k)
                        mma_ts(pv_o, d_s + 8 * k, dv + (uint64_t)(2 * D * k), C::kIdescPV,
                               (pv_acc || k > 0) ? 1u : 0u);
                    mma_commit(sready_s + 8u);
                }
            }
            __syncwarp();
            pv_owed = false;
        }
    } else if (warp < kFirstSoftmaxWarp) {
        // ------------------------------------------------------------ TMA producer
        // Order: A(0) .. A(kAAhead - 1), items(0), A(kAAhead), items(1), A(kAAhead + 1), ...
        // The A group of unit k goes into shared buffer k % kABufS once the group before it in
        // that buffer has been read by the last S product of its unit, which each softmax
        // warpgroup reports when it sees that S. Every wait blocks (try_wait), so the warp takes
        // no issue slots while it waits.
        regs_lower<kRegsControl>();
        if (warp == kProducerWarp) {
            const int64_t G = gridDim.x;
            uint32_t it = 0, na = 0;  // ring items and A groups issued
            int64_t withheld = -1;
            bool ok = true;
            auto issue_a = [&](uint32_t k, int64_t u) -> bool {
                const int ab = k % C::kABufS;
                if (!warp_wait(afree0 + 8u * ab,
                               ((k / C::kABufS) & 1) ^ 1, abort_flag, prm.status, prm.wait_ns))
                    return false;
                const Unit UA = get_unit<D, DEC, LO>(prm, u);
                if (elect_one()) {
                    mbar_expect_tx(afull0 + 8u * ab, UA.n_a * C::kANum * C::kATile);
                    for (int a = 0; a < UA.n_a; ++a) {
                        uint8_t* dst = abuf + ab * C::kABytes + a * C::kANum * C::kATile;
                        tma_load_3d(smem_u32(dst), &tmA, 0, UA.rowA0 + a * kTileRows, UA.zA,
                                    afull0 + 8u * ab);
                        if constexpr (C::kLoA)
                            tma_load_3d(smem_u32(dst + C::kATile), &tmL, 0,
                                        UA.rowA0 + a * kTileRows, UA.zA, afull0 + 8u * ab);
                    }
                }
                __syncwarp();
                ++na;
                return true;
            };
            for (uint32_t k = 0; k < (uint32_t)C::kAAhead && ok; ++k)
                if (blockIdx.x + k * G < prm.n_units) ok = issue_a(k, blockIdx.x + k * G);
            uint32_t k = 0;
            for (int64_t u = blockIdx.x; u < prm.n_units && ok; u += G, ++k) {
                const Unit U = get_unit<D, DEC, LO>(prm, u);
                for (int i = 0; i < U.n_items; ++i, ++it) {
                    const int st = it % C::kStages;
                    if (!warp_wait(empty0 + 8u * st, ((it / C::kStages) & 1) ^ 1, abort_flag,
                                   prm.status, prm.wait_ns)) {
                        ok = false;
                        break;
                    }
                    if (blockIdx.x == 0 && (int64_t)it == prm.withhold_it) {
                        withheld = it;  // never loaded: the waits of its consumers run out
                        continue;
                    }
                    if (elect_one()) {
                        mbar_expect_tx(full0 + 8u * st, C::kStage);
                        const int row = (int)(U.item0 + (int64_t)i * C::kItem);
                        const uint32_t dst = smem_u32(ring + st * C::kStage);
                        tma_load_3d(dst, &tmB, 0, row, U.zB, full0 + 8u * st);
                        tma_load_3d(dst + C::kItemTile, &tmC, 0, row, U.zB, full0 + 8u * st);
                        if constexpr (C::kLoB)
                            tma_load_3d(dst + 2 * C::kItemTile, &tmL, 0, row, U.zB,
                                        full0 + 8u * st);
                        // streams that do not take this item count as having released it
                        for (int x = U.n_a; x < NS; ++x) mbar_arrive(empty0 + 8u * st);
                    }
                    __syncwarp();
                }
                const int64_t un = u + C::kAAhead * G;
                if (ok && un < prm.n_units) ok = issue_a(k + C::kAAhead, un);
            }
            if (!ok) {
                // after an abort: wait (bounded) until the newest copy into every buffer landed
                const uint64_t t0 = globaltimer_ns();
                for (uint32_t st = 0; st < (uint32_t)C::kStages && st < it; ++st) {
                    const uint32_t x = it - 1 - ((it - 1 - st) % C::kStages);
                    while ((int64_t)x != withheld &&
                           !mbar_try_wait(full0 + 8u * st, (x / C::kStages) & 1) &&
                           globaltimer_ns() - t0 < prm.wait_ns) {
                    }
                }
                for (uint32_t b = 0; b < (uint32_t)C::kABufS && b < na; ++b) {
                    const uint32_t y = na - 1 - ((na - 1 - b) % C::kABufS);
                    while (!mbar_try_wait(afull0 + 8u * b, (y / C::kABufS) & 1) &&
                           globaltimer_ns() - t0 < prm.wait_ns) {
                    }
                }
            }
        }
    } else {
        // ------------------------------------------------------------ softmax warpgroups
        regs_raise<kRegsSoftmax>();
        const int wg = (warp - kFirstSoftmaxWarp) >> 2;
        const int q = warp & 3;
        const int r = q * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
        const bool wg_leader = ((warp - kFirstSoftmaxWarp) & 3) == 0 && lane == 0;
        const float c = prm.c;
        const uint64_t c2 = pack_f32x2(c, c);
        SoftmaxStream st;
        st.s = wg;
        st.ph0 = 0;
        st.od = 0;
        st.over = false;
        const uint32_t sready_s = sready0 + 16u * wg;
        bool alive = true;
        uint32_t ua = 0, it0 = 0;
        // With two O accumulators (decode) the end of a unit (reading O, the stores) runs after
        // the next unit's first item, whose s_ready also covers the unit's last PV, so it
        // overlaps that item's round trip to the MMA warp. Every decode unit gives every stream
        // all of its items (at least one), so that first item always exists.
        bool owed = false;
        UnitEnd prev{};
        for (int64_t u = blockIdx.x; u < prm.n_units && alive; u += gridDim.x, ++ua) {
            const Unit U = get_unit<D, DEC, LO>(prm, u);
            st.begin(U);
            st.ob = C::kOBuf == 2 ? (int)(ua & 1) : 0;
            st.ab = (int)(ua % C::kABufS);
            while (alive && st.j < st.cnt) {
                alive = softmax_step<D, DEC, SAFE, LO>(st, U, tmem, lane_off, c, c2, sready_s,
                                                   pready0 + 16u * st.s, empty0, afree0,
                                                   wg_leader, it0, abort_flag, prm.status,
                                                   prm.wait_ns, prm.overflow);
                if (owed && alive) {
                    alive = finish_stream<D, DEC, LO>(st, prev,
                                                      get_unit<D, DEC, LO>(prm, u - gridDim.x),
                                                      prm, tmem, lane_off, r, sready_s, empty0,
                                                      afree0, wg_leader, true, abort_flag);
                    owed = false;
                }
            }
            if (alive) {
                const UnitEnd e{st.m, st.l, st.cnt, st.ob, st.ab, it0};
                if (C::kOBuf == 2 && u + gridDim.x < prm.n_units) {
                    prev = e;
                    owed = true;
                } else {
                    alive = finish_stream<D, DEC, LO>(st, e, U, prm, tmem, lane_off, r, sready_s,
                                                      empty0, afree0, wg_leader, false, abort_flag);
                }
            }
            st.ph0 += (uint32_t)st.cnt;
            it0 += U.n_items;
        }
        if (!SAFE && __any_sync(0xffffffffu, st.over) && lane == 0) *prm.overflow = 1;
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ------------------------------------------------------------------ host side

// The test hook's setting (set_tc_test_fault): the launch it applies to (0: none; 1, 2: the
// encode of call 1 or 2; 3: the decode), the ring item withheld in CTA 0 and the wait bound
// of that launch.
struct TestFault {
    int kernel = 0;
    int64_t ring_item = -1;
    uint64_t wait_ns = kDefaultWaitNs;
};
std::mutex g_fault_mu;
TestFault g_fault;

void apply_fault(int kernel, TcParams& prm) {
    std::lock_guard<std::mutex> lock(g_fault_mu);
    prm.wait_ns = kDefaultWaitNs;
    prm.withhold_it = -1;
    if (g_fault.kernel != 0 && g_fault.kernel == kernel) {
        prm.wait_ns = g_fault.wait_ns;
        prm.withhold_it = g_fault.ring_item;
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        cudaDriverEntryPointQueryResult q;
        void* p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// 3D bf16 map over [z, rows, D] (D innermost) with a box of box_rows x D, swizzled to match
// one D-wide row (the layout the MMA descriptors of every operand tile assume).
bool make_map(CUtensorMap* m, const void* base, int64_t D, int64_t rows, int64_t z,
              uint32_t box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)rows, (cuuint64_t)z};
    cuuint64_t strides[2] = {(cuuint64_t)(D * 2), (cuuint64_t)(rows * D * 2)};
    cuuint32_t box[3] = {(cuuint32_t)D, box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    const CUtensorMapSwizzle sw =
        D == 16 ? CU_TENSOR_MAP_SWIZZLE_32B
                : (D == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B);
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The fast kernel, then the safe one on the same stream (it returns at once unless the
// fast kernel raised the overflow word, which the plan keeps zeroed before each call).
template <int D, bool DEC, bool LO>
cudaError_t launch(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                   const CUtensorMap& l, const TcParams& prm, cudaStream_t st) {
    using Cf = Cfg<D, DEC, LO>;
    cudaError_t e = ensure_smem_limit((const void*)tc_chain_kernel<D, DEC, false, LO>, Cf::kSmem);
    if (e == cudaSuccess)
        e = ensure_smem_limit((const void*)tc_chain_kernel<D, DEC, true, LO>, Cf::kSmem);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = kNumSMs;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t grid = prm.n_units < sms ? prm.n_units : sms;
    e = launch_pdl(tc_chain_kernel<D, DEC, false, LO>, dim3((unsigned)grid), dim3(kThreads),
                   Cf::kSmem, st, a, b, c, l, prm);
    if (e == cudaSuccess)
        e = launch_pdl(tc_chain_kernel<D, DEC, true, LO>, dim3((unsigned)grid), dim3(kThreads),
                       Cf::kSmem, st, a, b, c, l, prm);
    return e;
}

// `l` (the map of Q's lo tiles) is read only by the LO kernels (D <= 32).
template <bool DEC>
cudaError_t launch_d(int64_t D, bool lo, const CUtensorMap& a, const CUtensorMap& b,
                     const CUtensorMap& c, const CUtensorMap& l, const TcParams& prm,
                     cudaStream_t st) {
    if (lo) {
        switch (D) {
            case 16: return launch<16, DEC, true>(a, b, c, l, prm, st);
            case 32: return launch<32, DEC, true>(a, b, c, l, prm, st);
        }
        return cudaErrorInvalidValue;
    }
    switch (D) {
        case 16: return launch<16, DEC, false>(a, b, c, l, prm, st);
        case 32: return launch<32, DEC, false>(a, b, c, l, prm, st);
        case 64: return launch<64, DEC, false>(a, b, c, l, prm, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace

// Streamed rows per item (the TMA box height of the ring tiles) of the encode or decode.
template <bool DEC>
uint32_t item_rows(int64_t D, bool lo = false) {
    if (lo) return D == 16 ? Cfg<16, DEC, true>::kItem : Cfg<32, DEC, true>::kItem;
    return D == 16 ? Cfg<16, DEC>::kItem : (D == 32 ? Cfg<32, DEC>::kItem : Cfg<64, DEC>::kItem);
}

int64_t tc_encode_item_rows(int64_t D) { return item_rows<false>(D); }

void test_fault_for(int kernel, uint64_t* wait_ns, int64_t* ring_item) {
    std::lock_guard<std::mutex> lock(g_fault_mu);
    *wait_ns = kDefaultWaitNs;
    *ring_item = -1;
    if (g_fault.kernel != 0 && g_fault.kernel == kernel) {
        *wait_ns = g_fault.wait_ns;
        *ring_item = g_fault.ring_item;
    }
}

void set_tc_test_fault(int kernel, int64_t ring_item, uint64_t wait_ns) {
    std::lock_guard<std::mutex> lock(g_fault_mu);
    g_fault.kernel = kernel;
    g_fault.ring_item = ring_item;
    g_fault.wait_ns = wait_ns > 0 ? wait_ns : kDefaultWaitNs;
}

int64_t tc_group_rows(int64_t D) {
    (void)D;
    return NS * kTileRows;
}

cudaError_t tc_encode(const Plan& p, int call, const void* k, const void* v, const void* seeds,
                      float scale, char* ws, cudaStream_t st, bool lo) {
    CUtensorMap ma, mb, mc, ml;
    const bool neg = scale < 0.f;
    lo = lo && call == 2 && p.D <= 32;  // call 1's A operand (the seeds) is exact in bf16
    const void* a_src;
    int64_t a_z;
    if (call == 1) {
        a_src = neg ? (const void*)(ws + p.off_seedneg) : seeds;
        a_z = p.H;
    } else {
        a_src = ws + p.off_qop;
        a_z = p.BH;
    }
    if (!make_map(&ma, a_src, p.D, p.M, a_z, kTileRows) ||
        !make_map(&mb, k, p.D, p.N, p.BH, item_rows<false>(p.D, lo)) ||
        !make_map(&mc, v, p.D, p.N, p.BH, item_rows<false>(p.D, lo)))
        return cudaErrorInvalidValue;
    ml = ma;
    if (lo && !make_map(&ml, ws + p.off_qlo, p.D, p.M, a_z, kTileRows))
        return cudaErrorInvalidValue;
    TcParams prm{};
    prm.BH = p.BH;
    prm.H = p.H;
    prm.N = p.N;
    prm.M = p.M;
    prm.a_per_head = call == 1 ? 1 : 0;
    prm.c = fabsf(scale) * kLog2e;
    prm.chunk_len = p.chunk_len;
    prm.nchunk = p.nchunk;
    prm.n_groups = p.n_groups;
    prm.pmax = (float*)(ws + p.off_pmax);
    prm.psum = (float*)(ws + p.off_psum);
    prm.pacc = (float*)(ws + p.off_pacc);
    prm.n_units = p.BH * p.n_groups * p.nchunk;
    prm.status = (int*)(ws + p.off_status);
    prm.overflow = (int*)(ws + p.off_overflow) + (call - 1);
    apply_fault(call, prm);
    return launch_d<false>(p.D, lo, ma, mb, mc, ml, prm, st);
}

cudaError_t tc_decode(const Plan& p, const void* K, float scale, void* Y, char* ws,
                      cudaStream_t st, float* lse, bool lo) {
    CUtensorMap ma, mb, mc, ml;
    lo = lo && p.D <= 32;
    if (!make_map(&ma, K, p.D, p.N, p.BH, kTileRows) ||
        !make_map(&mb, ws + p.off_qop, p.D, p.M, p.BH, item_rows<true>(p.D, lo)) ||
        !make_map(&mc, ws + p.off_zop, p.D, p.M, p.BH, item_rows<true>(p.D, lo)))
        return cudaErrorInvalidValue;
    ml = ma;
    if (lo && !make_map(&ml, ws + p.off_qlo, p.D, p.M, p.BH, item_rows<true>(p.D, lo)))
        return cudaErrorInvalidValue;
    TcParams prm{};
    prm.BH = p.BH;
    prm.H = p.H;
    prm.N = p.N;
    prm.M = p.M;
    prm.c = fabsf(scale) * kLog2e;
    const int64_t grp = tc_group_rows(p.D);
    prm.n_tok_groups = (p.N + grp - 1) / grp;
    prm.Y = (__nv_bfloat16*)Y;
    prm.lse = lse;
    prm.n_units = p.BH * prm.n_tok_groups;
    prm.status = (int*)(ws + p.off_status);
    prm.overflow = (int*)(ws + p.off_overflow) + 2;
    apply_fault(3, prm);
    return launch_d<true>(p.D, lo, ma, mb, mc, ml, prm, st);
}

}  // namespace flarepp
