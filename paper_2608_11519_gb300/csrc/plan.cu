// The shape-derived plan of a call: which kernels run, how the tokens are cut into chunks
// for the split-N encode (App. A.2), and the workspace layout. The plan fixes every launch
// configuration, so this file and the kernel sources together determine what each kernel
// reads and writes.
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include "flarepp_internal.h"

namespace flarepp {
namespace {

constexpr int64_t kMaxM = 2048;
constexpr int64_t kMaxTokenHeads = int64_t(1) << 40;  // B*H*N limit (index headroom)
constexpr int64_t kMaxTmaCoord = 2147483647 - 4096;  // TMA coordinates are signed 32-bit

bool mul_ok(int64_t a, int64_t b, int64_t* out) { return !__builtin_mul_overflow(a, b, out); }

}  // namespace

flarepp_status make_plan(const flarepp_shape* s, Plan* p) {
    if (!s || !p) return FLAREPP_ERR_INVALID_ARGUMENT;
    if (s->dtype != FLAREPP_F32 && s->dtype != FLAREPP_BF16) return FLAREPP_ERR_INVALID_ARGUMENT;
    if (s->B < 0 || s->H < 0 || s->N < 0 || s->M < 0 || s->D < 0)
        return FLAREPP_ERR_INVALID_ARGUMENT;
    if (s->D != 16 && s->D != 32 && s->D != 64) return FLAREPP_ERR_UNSUPPORTED;
    if (s->M > kMaxM) return FLAREPP_ERR_UNSUPPORTED;
    int64_t bh, bhn;
    if (!mul_ok(s->B, s->H, &bh) || !mul_ok(bh, s->N, &bhn)) return FLAREPP_ERR_UNSUPPORTED;
    if (bhn > kMaxTokenHeads) return FLAREPP_ERR_UNSUPPORTED;

    memset(p, 0, sizeof(*p));
    p->B = s->B;
    p->H = s->H;
    p->N = s->N;
    p->M = s->M;
    p->D = s->D;
    p->BH = bh;
    p->dtype = s->dtype;
    p->path = s->dtype == FLAREPP_BF16 ? kPathTc : kPathSimt;
    if (p->path == kPathTc && (s->N > kMaxTmaCoord || bh > kMaxTmaCoord))
        return FLAREPP_ERR_UNSUPPORTED;
    if (bh == 0 || s->N == 0 || s->M == 0) return FLAREPP_OK;  // nothing to plan

    if (p->path == kPathSimt) {
        // CUDA-core encode: one thread per route, up to 128 routes per CTA; chunks sized so
        // that the grid holds about four waves of CTAs per SM.
        p->m_tile = s->M >= 128 ? 128 : cdiv(s->M, 32) * 32;
        p->n_mtiles = cdiv(s->M, p->m_tile);
        p->sub_per_chunk = 1;
        const int64_t target = 4 * kNumSMs;
        int64_t want = cdiv(target, bh * p->n_mtiles);
        if (want < 1) want = 1;
        p->chunk_len = cdiv(cdiv(s->N, want), 32) * 32;
        p->nchunk = cdiv(s->N, p->chunk_len);
    } else {
        // Tensor-core encode: a work unit is (bh, group of <= 512 routes, chunk of tokens) and
        // one persistent CTA per SM walks the units. Pick the chunk count that minimises
        // waves x (items per unit, scaled by the group's route tiles, + a fixed per-unit
        // cost of about three items); chunks are whole items.
        p->tc_group = tc_group_rows(s->D);
        const int64_t kTcItem = tc_encode_item_rows(s->D);  // tokens per encode item
        p->n_groups = cdiv(s->M, p->tc_group);
        p->sub_per_chunk = 4;
        const int64_t ns = p->tc_group / 128;
        const int64_t tiles0 = s->M >= p->tc_group ? ns : cdiv(s->M, 128);
        const double na = tiles0 <= 1 ? 1.0 : (tiles0 <= 2 ? 2.0 : 4.0);
        const int64_t per_chunk = bh * p->n_groups;
        // The waves grow with n and the items per unit shrink, so among the chunk counts
        // with the same number of waves the largest costs least: only that one is tried for
        // each wave count. For every n, waves x items >= per_chunk * N / (SMs * item), so
        // the cost is at least that product's share plus 3 x waves; once this bound reaches
        // the best cost found, no larger count can win and the search stops. This finds the
        // same chunk length as trying every count from 1 (ties within one wave count have
        // equal items), in far fewer steps.
        const int64_t max_chunks = cdiv(s->N, kTcItem);
        const int64_t cap = max_chunks < 65536 ? max_chunks : 65536;
        const double floor_items = 0.999999 * (double)per_chunk * (double)s->N * na /
                                   ((double)kNumSMs * (double)kTcItem * (double)ns);
        double best = 1e300;
        int64_t best_n = 1;
        for (int64_t n = 1; n <= cap;) {
            const int64_t waves = cdiv(per_chunk * n, kNumSMs);
            if (floor_items + 3.0 * (double)waves >= best) break;
            int64_t hi = waves * kNumSMs / per_chunk;  // the largest count with these waves
            if (hi > cap) hi = cap;
            const int64_t items = cdiv(cdiv(s->N, hi), kTcItem);
            const double cost = (double)waves * ((double)items * na / (double)ns + 3.0);
            if (cost < best) {
                best = cost;
                best_n = hi;
            }
            n = hi + 1;
        }
        p->chunk_len = cdiv(cdiv(s->N, best_n), kTcItem) * kTcItem;
        p->nchunk = cdiv(s->N, p->chunk_len);
        // the kernels count their work units in 32 bits
        if (per_chunk * p->nchunk > INT32_MAX || bh * cdiv(s->N, p->tc_group) > INT32_MAX)
            return FLAREPP_ERR_UNSUPPORTED;
    }

    const size_t rows =
        (size_t)bh * (size_t)p->nchunk * (size_t)p->sub_per_chunk * (size_t)s->M;
    size_t off = 0;
    p->off_status = off;
    // the overflow words of encode calls 1 and 2 and of the decode (tensor-core path) share
    // the status word's 256-byte block
    p->off_overflow = off + 16;
    off = align_up(off + 16 + 3 * sizeof(int32_t), kWsAlign);
    p->off_pmax = off;
    off = align_up(off + rows * sizeof(float), kWsAlign);
    p->off_psum = off;
    off = align_up(off + rows * sizeof(float), kWsAlign);
    p->off_pacc = off;
    off = align_up(off + rows * (size_t)s->D * sizeof(float), kWsAlign);
    const size_t qz = (size_t)bh * (size_t)s->M * (size_t)s->D * sizeof(float);
    p->off_q32 = off;
    off = align_up(off + qz, kWsAlign);
    p->off_z32 = off;
    off = align_up(off + qz, kWsAlign);
    if (p->path == kPathTc) {
        const size_t op = (size_t)bh * (size_t)s->M * (size_t)s->D * 2;
        p->off_qop = off;
        off = align_up(off + op, kWsAlign);
        p->off_zop = off;
        off = align_up(off + op, kWsAlign);
        p->off_qlo = off;
        off = align_up(off + op, kWsAlign);
        p->off_seedneg = off;
        off = align_up(off + (size_t)s->H * (size_t)s->M * (size_t)s->D * 2, kWsAlign);
    }
    p->total = off;
    return FLAREPP_OK;
}

SavedLayout saved_layout(const Plan& p) {
    SavedLayout L{};
    const size_t qz = (size_t)p.BH * (size_t)p.M * (size_t)p.D * sizeof(float);
    const size_t lm = (size_t)p.BH * (size_t)p.M * sizeof(float);
    const size_t ln = (size_t)p.BH * (size_t)p.N * sizeof(float);
    size_t off = 0;
    L.off_q = off;
    off = align_up(off + qz, kWsAlign);
    L.off_z = off;
    off = align_up(off + qz, kWsAlign);
    L.off_l1 = off;
    off = align_up(off + lm, kWsAlign);
    L.off_l2 = off;
    off = align_up(off + lm, kWsAlign);
    L.off_l3 = off;
    off = align_up(off + ln, kWsAlign);
    L.total = off;
    return L;
}

BwdPlan make_bwd_plan(const Plan& p) {
    BwdPlan b{};
    b.path = p.path;
    if (p.BH == 0 || p.N == 0 || p.M == 0) return b;
    b.m_tile = p.M >= 128 ? 128 : cdiv(p.M, 32) * 32;
    b.n_mtiles = cdiv(p.M, b.m_tile);
    if (p.path == kPathTc) {
        // work units (b*h, route group of up to 512, chunk): about two waves of persistent
        // CTAs; chunks are whole items (192 tokens is a multiple of every item size)
        const int64_t item = 192;
        const int64_t groups = cdiv(p.M, 512);
        int64_t want = cdiv(2 * kNumSMs, p.BH * groups);
        if (want < 1) want = 1;
        b.chunk_len = cdiv(cdiv(p.N, want), item) * item;
    } else {
        // one thread per route, up to 128 routes per CTA; chunks for about four waves
        int64_t want = cdiv(4 * kNumSMs, p.BH * b.n_mtiles);
        if (want < 1) want = 1;
        b.chunk_len = cdiv(cdiv(p.N, want), 32) * 32;
    }
    b.nchunk = cdiv(p.N, b.chunk_len);
    const size_t part = (size_t)p.BH * (size_t)b.nchunk * (size_t)p.M * (size_t)p.D * 4;
    const size_t qz = (size_t)p.BH * (size_t)p.M * (size_t)p.D * 4;
    const size_t lm = (size_t)p.BH * (size_t)p.M * 4;
    const size_t ln = (size_t)p.BH * (size_t)p.N * 4;
    size_t off = 0;
    b.off_status = off;
    off = align_up(off + sizeof(int32_t), kWsAlign);
    b.off_pa = off;
    off = align_up(off + part, kWsAlign);
    b.off_pb = off;
    off = align_up(off + part, kWsAlign);
    b.off_dz = off;
    off = align_up(off + qz, kWsAlign);
    b.off_dq = off;
    off = align_up(off + qz, kWsAlign);
    b.off_d1 = off;
    off = align_up(off + lm, kWsAlign);
    b.off_d2 = off;
    off = align_up(off + lm, kWsAlign);
    b.off_d3 = off;
    off = align_up(off + ln + 256, kWsAlign);
    if (p.path == kPathTc) {
        const size_t op = (size_t)p.BH * (size_t)p.M * (size_t)p.D * 2;
        b.off_qb = off;
        off = align_up(off + op, kWsAlign);
        b.off_zb = off;
        off = align_up(off + op, kWsAlign);
        b.off_dzb = off;
        off = align_up(off + op, kWsAlign);
        b.off_dqb = off;
        off = align_up(off + op, kWsAlign);
        b.off_qlo = off;
        off = align_up(off + op, kWsAlign);
        b.off_w = off;
        off = align_up(off + op, kWsAlign);
        b.off_rb = off;
        off = align_up(off + (size_t)p.BH * 4, kWsAlign);
        b.off_flags = off;
        off = align_up(off + (size_t)p.BH * 4, kWsAlign);
        b.off_rpart = off;
        off = align_up(off + (size_t)p.BH * (kRangeParts + 2) * 4, kWsAlign);
    }
    b.total = off;
    return b;
}

}  // namespace flarepp
