// Tensor-core (tcgen05 / TMEM / TMA) kernels of the routing chain: the bf16 dtype path.
//
// One warp-specialised kernel template serves both directions of the routing chain
// (Sec. 3.2, eqs. flarepp_dynamic_query and flarepp_mixer):
//
//   encode (calls 1, 2): TMEM lanes are routes. A resident group of up to 4 route tiles
//     (128 routes each, the A operand: seeds or Q) meets a stream of 64-token items
//     (K and V tiles) from a chunk of the sequence; each route row keeps an online
//     softmax over tokens and the CTA writes per-chunk partials (running max, sum and
//     unnormalised value sum) for the log-sum-exp merge of App. A.3.
//   decode (call 3): TMEM lanes are tokens. A resident group of 4 token tiles (K, 128
//     tokens each) meets a stream of 64-route items (Q and Z tiles); each token row keeps
//     an online softmax over routes and writes its normalised output row of Y.
//
// Roles (10 warps): warp 0 issues TMA loads, warp 1 issues tcgen05.mma (one thread) and
// owns the TMEM allocation, warps 2-9 form two softmax warpgroups. The four TMEM
// "streams" s = 0..3 each hold a 128 x 64 fp32 score tile S (reused in place for the
// bf16 probabilities P, the A operand of the PV product) and a 128 x D fp32 accumulator
// O; warpgroup w serves streams w and w + 2. Per stream and item:
//   MMA warp: S = A_tile * B_item^T (K-major, smem x smem) -> commit s_ready
//   softmax:  row max, lazily raised running max (rescaling O in TMEM only when the max
//             grows by more than 2^8), P = 2^(c S - m) in bf16 back into TMEM, row sum
//             -> arrive p_ready
//   MMA warp: O += P * C_item (P from TMEM, C MN-major in smem); the next S of the stream
//             is issued after it, so a completed s_ready also means the previous PV is done.
// Every wait is bounded (2 s of %globaltimer): on expiry the kernel records
// FLAREPP_ERR_TIMEOUT in the status word, all roles leave their loops, and TMEM is freed.
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

constexpr int kThreads = 320;
constexpr int kTileRows = 128;
constexpr int kItem = 64;          // streamed rows per item
constexpr int kGroup = 512;        // resident rows per work unit (4 tiles of 128)
constexpr float kLazyTau = 8.0f;   // log2 headroom of the lazy running max
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint32_t kTmemCols = 512;
constexpr float kLog2e = 1.4426950408889634f;

template <int D>
struct Cfg {
    static constexpr int kStages = D == 64 ? 5 : 8;
    static constexpr int kATile = kTileRows * D * 2;
    static constexpr int kABytes = 4 * kATile;
    static constexpr int kItemTile = kItem * D * 2;
    static constexpr int kStage = 2 * kItemTile;
    static constexpr uint32_t kSwz = D == 16 ? kSw32 : (D == 32 ? kSw64 : kSw128);
    static constexpr uint32_t kSBO = 8 * D * 2;
    static constexpr int kNumBars = 2 * kStages + 12;
    static constexpr int kData = 2 * kABytes + kStages * kStage;
    static constexpr int kNeed = 1024 + kData + kNumBars * 8 + 16;
    // at least 120 KB so that one CTA owns an SM and its 512 TMEM columns
    static constexpr int kSmem = kNeed > 122880 ? kNeed : 122880;
    static constexpr uint32_t kIdescS = idesc_bf16_f32(128, kItem, false, false);
    static constexpr uint32_t kIdescPV = idesc_bf16_f32(128, D, false, true);
    static constexpr uint32_t kOCol = 4 * kItem;  // O accumulators follow the 4 score tiles
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
    int64_t n_units;
    int* status;
};

__device__ __forceinline__ int na_of_group(int64_t M, int64_t g) {
    const int64_t rem = M - g * kGroup;
    const int64_t tiles = rem >= kGroup ? 4 : (rem + kTileRows - 1) / kTileRows;
    return tiles <= 1 ? 1 : (tiles <= 2 ? 2 : 4);
}

struct Unit {
    int64_t bh, chunk, g, tg;
    int zA, rowA0, zB;
    int n_a, n_par, n_items;
    int64_t item0, item_end;
};

template <bool DEC>
__device__ __forceinline__ Unit get_unit(const TcParams& p, int64_t u) {
    Unit U;
    if (DEC) {
        U.tg = u % p.n_tok_groups;
        U.bh = u / p.n_tok_groups;
        U.chunk = 0;
        U.g = 0;
        U.zA = (int)U.bh;
        U.rowA0 = (int)(U.tg * kGroup);
        U.n_a = 4;
        U.n_par = 1;
        U.item0 = 0;
        U.item_end = p.M;
    } else {
        U.chunk = u % p.nchunk;
        const int64_t t = u / p.nchunk;
        U.g = t % p.n_groups;
        U.bh = t / p.n_groups;
        U.tg = 0;
        U.zA = (int)(p.a_per_head ? U.bh % p.H : U.bh);
        U.rowA0 = (int)(U.g * kGroup);
        U.n_a = na_of_group(p.M, U.g);
        U.n_par = 4 / U.n_a;
        U.item0 = U.chunk * p.chunk_len;
        U.item_end = min(p.N, U.item0 + p.chunk_len);
    }
    U.zB = (int)U.bh;
    U.n_items = (int)((U.item_end - U.item0 + kItem - 1) / kItem);
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

template <int D, bool DEC>
__global__ void __launch_bounds__(kThreads, 1)
    tc_chain_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmC, const TcParams prm) {
    using C = Cfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    uint8_t* abuf = smem;
    uint8_t* ring = smem + 2 * C::kABytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(ring + C::kStages * C::kStage);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::kNumBars);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int st) { return bar0 + 8u * st; };
    auto empty_bar = [&](int st) { return bar0 + 8u * (C::kStages + st); };
    auto afull_bar = [&](int b) { return bar0 + 8u * (2 * C::kStages + b); };
    auto aempty_bar = [&](int b) { return bar0 + 8u * (2 * C::kStages + 2 + b); };
    auto sready_bar = [&](int s) { return bar0 + 8u * (2 * C::kStages + 4 + s); };
    auto pready_bar = [&](int s) { return bar0 + 8u * (2 * C::kStages + 8 + s); };

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int st = 0; st < C::kStages; ++st) {
            mbar_init(full_bar(st), 1);
            mbar_init(empty_bar(st), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(afull_bar(b), 1);
            mbar_init(aempty_bar(b), 1);
        }
        for (int s = 0; s < 4; ++s) {
            mbar_init(sready_bar(s), 1);
            mbar_init(pready_bar(s), 128);
        }
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmA);
        prefetch_tmap(&tmB);
        prefetch_tmap(&tmC);
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
        if (lane == 0) {
            uint32_t it = 0, ua = 0;
            for (int64_t u = blockIdx.x; u < prm.n_units; u += gridDim.x) {
                const Unit U = get_unit<DEC>(prm, u);
                const int ab = ua & 1;
                if (!wait_bar(aempty_bar(ab), ((ua >> 1) & 1) ^ 1, abort_flag, prm.status)) break;
                mbar_expect_tx(afull_bar(ab), U.n_a * C::kATile);
                for (int a = 0; a < U.n_a; ++a)
                    tma_load_3d(smem_u32(abuf + ab * C::kABytes + a * C::kATile), &tmA, 0,
                                U.rowA0 + a * kTileRows, U.zA, afull_bar(ab));
                ++ua;
                bool ok = true;
                for (int i = 0; i < U.n_items; ++i) {
                    const int st = it % C::kStages;
                    if (!wait_bar(empty_bar(st), ((it / C::kStages) & 1) ^ 1, abort_flag,
                                  prm.status)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(full_bar(st), C::kStage);
                    const int row = (int)(U.item0 + (int64_t)i * kItem);
                    const uint32_t dst = smem_u32(ring + st * C::kStage);
                    tma_load_3d(dst, &tmB, 0, row, U.zB, full_bar(st));
                    tma_load_3d(dst + C::kItemTile, &tmC, 0, row, U.zB, full_bar(st));
                    ++it;
                }
                if (!ok) break;
            }
            if (*abort_flag) {
                // Leave only after every copy this thread issued has landed: the newest load
                // of each stage and of each A buffer (older ones were consumed already).
                const uint64_t t0 = globaltimer_ns();
                for (int st = 0; st < C::kStages; ++st) {
                    if ((uint32_t)st >= it) break;
                    const uint32_t x = it - 1 - ((it - 1 - st) % C::kStages);
                    while (!mbar_try_wait(full_bar(st), (x / C::kStages) & 1) &&
                           globaltimer_ns() - t0 < kWaitLimitNs) {
                    }
                }
                for (int b = 0; b < 2; ++b) {
                    if ((uint32_t)b >= ua) break;
                    const uint32_t y = ua - 1 - ((ua - 1 - b) % 2);
                    while (!mbar_try_wait(afull_bar(b), (y >> 1) & 1) &&
                           globaltimer_ns() - t0 < kWaitLimitNs) {
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            uint32_t it = 0, ua = 0;
            uint32_t pcnt[4] = {0, 0, 0, 0};
            bool ok = true;
            for (int64_t u = blockIdx.x; u < prm.n_units && ok; u += gridDim.x, ++ua) {
                const Unit U = get_unit<DEC>(prm, u);
                const int ab = ua & 1;
                if (!wait_bar(afull_bar(ab), (ua >> 1) & 1, abort_flag, prm.status)) break;
                tc_fence_after();
                const uint32_t a_base = smem_u32(abuf + ab * C::kABytes);
                int prev_st[4] = {-1, -1, -1, -1};
                int npv[4] = {0, 0, 0, 0};
                int done[C::kStages];
#pragma unroll
                for (int st = 0; st < C::kStages; ++st) done[st] = 0;

                auto issue_pv = [&](int s) {
                    const uint32_t cb = smem_u32(ring + prev_st[s] * C::kStage + C::kItemTile);
#pragma unroll
                    for (int k = 0; k < kItem / 16; ++k) {
                        const uint64_t bd = smem_desc(cb + k * 16 * D * 2, C::kItemTile, C::kSBO,
                                                      C::kSwz);
                        mma_ts(tmem + C::kOCol + s * D, tmem + s * kItem + 8 * k, bd,
                               C::kIdescPV, (npv[s] > 0 || k > 0) ? 1u : 0u);
                    }
                    ++npv[s];
                    if (++done[prev_st[s]] == U.n_a) {
                        done[prev_st[s]] = 0;
                        mma_commit(empty_bar(prev_st[s]));
                    }
                };

                for (int i = 0; i < U.n_items && ok; ++i, ++it) {
                    const int st = it % C::kStages;
                    const uint32_t bb = smem_u32(ring + st * C::kStage);
                    bool have_item = false;
                    for (int a = 0; a < U.n_a; ++a) {
                        const int s = a + U.n_a * (i % U.n_par);
                        // the stream's previous PV first: it may free the stage item i needs
                        if (prev_st[s] >= 0) {
                            if (!wait_bar(pready_bar(s), pcnt[s] & 1, abort_flag, prm.status)) {
                                ok = false;
                                break;
                            }
                            ++pcnt[s];
                            tc_fence_after();
                            issue_pv(s);
                        }
                        if (!have_item) {
                            if (!wait_bar(full_bar(st), (it / C::kStages) & 1, abort_flag,
                                          prm.status)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            have_item = true;
                        }
                        const uint32_t ab_tile = a_base + a * C::kATile;
#pragma unroll
                        for (int k = 0; k < D / 16; ++k) {
                            const uint64_t ad = smem_desc(ab_tile + 32 * k, 16, C::kSBO, C::kSwz);
                            const uint64_t bd = smem_desc(bb + 32 * k, 16, C::kSBO, C::kSwz);
                            mma_ss(tmem + s * kItem, ad, bd, C::kIdescS, k > 0 ? 1u : 0u);
                        }
                        mma_commit(sready_bar(s));
                        prev_st[s] = st;
                    }
                }
                // drain: the last PV of every stream, then the final s_ready (O complete)
                for (int s = 0; s < 4 && ok; ++s) {
                    if (prev_st[s] < 0) continue;
                    if (!wait_bar(pready_bar(s), pcnt[s] & 1, abort_flag, prm.status)) {
                        ok = false;
                        break;
                    }
                    ++pcnt[s];
                    tc_fence_after();
                    issue_pv(s);
                    mma_commit(sready_bar(s));
                }
                mma_commit(aempty_bar(ab));
            }
        }
    } else {
        // ------------------------------------------------------------ softmax warpgroups
        const int wg = (warp - 2) >> 2;
        const int q = warp & 3;
        const int r = q * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
        const float c = prm.c;
        uint32_t scnt[2] = {0, 0};
        bool alive = true;
        for (int64_t u = blockIdx.x; u < prm.n_units && alive; u += gridDim.x) {
            const Unit U = get_unit<DEC>(prm, u);
            int cnt[2], sid[2];
            float m[2], l[2];
            int j[2] = {0, 0};
#pragma unroll
            for (int sl = 0; sl < 2; ++sl) {
                sid[sl] = wg + 2 * sl;
                const int par = sid[sl] / U.n_a;
                cnt[sl] = U.n_items > par ? (U.n_items - par + U.n_par - 1) / U.n_par : 0;
                m[sl] = -INFINITY;
                l[sl] = 0.f;
            }
            while (alive && (j[0] < cnt[0] || j[1] < cnt[1])) {
#pragma unroll
                for (int sl = 0; sl < 2; ++sl) {
                    if (j[sl] >= cnt[sl] || !alive) continue;
                    const int s = sid[sl];
                    const bool got = wait_bar(sready_bar(s), scnt[sl] & 1, abort_flag, prm.status);
                    ++scnt[sl];
                    if (!__all_sync(0xffffffffu, got)) {
                        alive = false;
                        continue;
                    }
                    tc_fence_after();
                    const int item = (s / U.n_a) + j[sl] * U.n_par;
                    const int64_t start = U.item0 + (int64_t)item * kItem;
                    const int nv = (int)min((int64_t)kItem, U.item_end - start);
                    const uint32_t scol = tmem + lane_off + s * kItem;
                    uint32_t sr[kItem];
#pragma unroll
                    for (int k = 0; k < kItem / 16; ++k) tmem_ld16(scol + 16 * k, sr + 16 * k);
                    tmem_wait_ld();
                    float mx;
                    if (nv == kItem) {
                        float a0 = __uint_as_float(sr[0]), a1 = __uint_as_float(sr[1]);
                        float a2 = __uint_as_float(sr[2]), a3 = __uint_as_float(sr[3]);
#pragma unroll
                        for (int k = 4; k < kItem; k += 4) {
                            a0 = fmaxf(a0, __uint_as_float(sr[k]));
                            a1 = fmaxf(a1, __uint_as_float(sr[k + 1]));
                            a2 = fmaxf(a2, __uint_as_float(sr[k + 2]));
                            a3 = fmaxf(a3, __uint_as_float(sr[k + 3]));
                        }
                        mx = fmaxf(fmaxf(a0, a1), fmaxf(a2, a3));
                    } else {
                        mx = -INFINITY;
#pragma unroll
                        for (int k = 0; k < kItem; ++k)
                            if (k < nv) mx = fmaxf(mx, __uint_as_float(sr[k]));
                    }
                    const float cand = mx * c;
                    bool need = false;
                    float alpha = 1.f;
                    if (cand > m[sl] + kLazyTau) {
                        alpha = ex2(m[sl] - cand);  // 0 on the first item
                        need = j[sl] > 0;
                        l[sl] *= alpha;
                        m[sl] = cand;
                    }
                    if (__any_sync(0xffffffffu, need)) {
                        const uint32_t ocol = tmem + lane_off + C::kOCol + s * D;
                        const float f = need ? alpha : 1.f;
#pragma unroll
                        for (int k = 0; k < D / 16; ++k) {
                            uint32_t o[16];
                            tmem_ld16(ocol + 16 * k, o);
                            tmem_wait_ld();
#pragma unroll
                            for (int e = 0; e < 16; ++e)
                                o[e] = __float_as_uint(__uint_as_float(o[e]) * f);
                            tmem_st16(ocol + 16 * k, o);
                        }
                    }
                    const float nm = -m[sl];
                    float sum0 = 0.f, sum1 = 0.f;
                    uint32_t pr[kItem / 2];
                    if (nv == kItem) {
#pragma unroll
                        for (int k = 0; k < kItem / 2; ++k) {
                            const float p0 = ex2(fmaf(__uint_as_float(sr[2 * k]), c, nm));
                            const float p1 = ex2(fmaf(__uint_as_float(sr[2 * k + 1]), c, nm));
                            sum0 += p0;
                            sum1 += p1;
                            pr[k] = pack_bf16(p0, p1);
                        }
                    } else {
#pragma unroll
                        for (int k = 0; k < kItem / 2; ++k) {
                            float p0 = ex2(fmaf(__uint_as_float(sr[2 * k]), c, nm));
                            float p1 = ex2(fmaf(__uint_as_float(sr[2 * k + 1]), c, nm));
                            p0 = (2 * k < nv) ? p0 : 0.f;
                            p1 = (2 * k + 1 < nv) ? p1 : 0.f;
                            sum0 += p0;
                            sum1 += p1;
                            pr[k] = pack_bf16(p0, p1);
                        }
                    }
                    l[sl] += sum0 + sum1;
                    tmem_st16(scol, pr);
                    tmem_st16(scol + 16, pr + 16);
                    tmem_wait_st();
                    tc_fence_before();
                    mbar_arrive(pready_bar(s));
                    ++j[sl];
                }
            }
            // results of the unit
#pragma unroll
            for (int sl = 0; sl < 2; ++sl) {
                if (!alive) break;
                const int s = sid[sl];
                const int a = s % U.n_a;
                const int par = s / U.n_a;
                float o[D];
                if (cnt[sl] > 0) {
                    const bool got = wait_bar(sready_bar(s), scnt[sl] & 1, abort_flag, prm.status);
                    ++scnt[sl];
                    if (!__all_sync(0xffffffffu, got)) {
                        alive = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t ocol = tmem + lane_off + C::kOCol + s * D;
#pragma unroll
                    for (int k = 0; k < D / 16; ++k) {
                        uint32_t t[16];
                        tmem_ld16(ocol + 16 * k, t);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 16; ++e) o[16 * k + e] = __uint_as_float(t[e]);
                    }
                } else {
#pragma unroll
                    for (int d = 0; d < D; ++d) o[d] = 0.f;
                }
                if (DEC) {
                    const int64_t tok = U.tg * kGroup + a * kTileRows + r;
                    if (tok < prm.N) {
                        const float inv = 1.f / l[sl];
                        uint4* dst = reinterpret_cast<uint4*>(prm.Y + (U.bh * prm.N + tok) * D);
#pragma unroll
                        for (int k = 0; k < D / 8; ++k) {
                            uint4 v;
                            v.x = pack_bf16(o[8 * k + 0] * inv, o[8 * k + 1] * inv);
                            v.y = pack_bf16(o[8 * k + 2] * inv, o[8 * k + 3] * inv);
                            v.z = pack_bf16(o[8 * k + 4] * inv, o[8 * k + 5] * inv);
                            v.w = pack_bf16(o[8 * k + 6] * inv, o[8 * k + 7] * inv);
                            dst[k] = v;
                        }
                    }
                } else {
                    const int64_t route = U.g * kGroup + a * kTileRows + r;
                    if (route < prm.M) {
                        const int64_t idx =
                            (U.bh * (prm.nchunk * 4) + U.chunk * 4 + par) * prm.M + route;
                        prm.pmax[idx] = cnt[sl] > 0 ? m[sl] : -INFINITY;
                        prm.psum[idx] = l[sl];
                        float4* dst = reinterpret_cast<float4*>(prm.pacc + idx * D);
#pragma unroll
                        for (int k = 0; k < D / 4; ++k)
                            dst[k] = make_float4(o[4 * k], o[4 * k + 1], o[4 * k + 2], o[4 * k + 3]);
                    }
                }
            }
        }
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

// 3D bf16 map over [z, rows, D] (D innermost) with a box of box_rows x D and the swizzle
// that matches one D-wide row.
bool make_map(CUtensorMap* m, const void* base, int64_t D, int64_t rows, int64_t z,
              uint32_t box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)rows, (cuuint64_t)z};
    cuuint64_t strides[2] = {(cuuint64_t)(D * 2), (cuuint64_t)(rows * D * 2)};
    cuuint32_t box[3] = {(cuuint32_t)D, box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    const CUtensorMapSwizzle sw = D == 16 ? CU_TENSOR_MAP_SWIZZLE_32B
                                  : D == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                            : CU_TENSOR_MAP_SWIZZLE_128B;
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D, bool DEC>
cudaError_t launch(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                   const TcParams& prm, cudaStream_t st) {
    using Cf = Cfg<D>;
    static cudaError_t attr = cudaFuncSetAttribute(
        tc_chain_kernel<D, DEC>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cf::kSmem);
    if (attr != cudaSuccess) return attr;
    int dev = 0, sms = kNumSMs;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t grid = prm.n_units < sms ? prm.n_units : sms;
    tc_chain_kernel<D, DEC><<<(unsigned)grid, kThreads, Cf::kSmem, st>>>(a, b, c, prm);
    return cudaGetLastError();
}

template <bool DEC>
cudaError_t launch_d(int64_t D, const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                     const TcParams& prm, cudaStream_t st) {
    switch (D) {
        case 16: return launch<16, DEC>(a, b, c, prm, st);
        case 32: return launch<32, DEC>(a, b, c, prm, st);
        case 64: return launch<64, DEC>(a, b, c, prm, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t tc_encode(const Plan& p, int call, const void* k, const void* v, const void* seeds,
                      float scale, char* ws, cudaStream_t st) {
    CUtensorMap ma, mb, mc;
    const bool neg = scale < 0.f;
    const void* a_src;
    int64_t a_z;
    if (call == 1) {
        a_src = neg ? (const void*)(ws + p.off_seedneg) : seeds;
        a_z = p.H;
    } else {
        a_src = ws + p.off_qop;
        a_z = p.BH;
    }
    if (!make_map(&ma, a_src, p.D, p.M, a_z, kTileRows) || !make_map(&mb, k, p.D, p.N, p.BH, kItem) ||
        !make_map(&mc, v, p.D, p.N, p.BH, kItem))
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
    return launch_d<false>(p.D, ma, mb, mc, prm, st);
}

cudaError_t tc_decode(const Plan& p, const void* K, float scale, void* Y, char* ws,
                      cudaStream_t st) {
    CUtensorMap ma, mb, mc;
    if (!make_map(&ma, K, p.D, p.N, p.BH, kTileRows) ||
        !make_map(&mb, ws + p.off_qop, p.D, p.M, p.BH, kItem) ||
        !make_map(&mc, ws + p.off_zop, p.D, p.M, p.BH, kItem))
        return cudaErrorInvalidValue;
    TcParams prm{};
    prm.BH = p.BH;
    prm.H = p.H;
    prm.N = p.N;
    prm.M = p.M;
    prm.c = fabsf(scale) * kLog2e;
    prm.n_tok_groups = (p.N + kGroup - 1) / kGroup;
    prm.Y = (__nv_bfloat16*)Y;
    prm.n_units = p.BH * prm.n_tok_groups;
    prm.status = (int*)(ws + p.off_status);
    return launch_d<true>(p.D, ma, mb, mc, prm, st);
}

}  // namespace flarepp
