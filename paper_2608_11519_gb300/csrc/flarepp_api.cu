// The C ABI of libflarepp: argument checks, the shape-derived plan and workspace layout,
// and the launch sequence of the routing chain (Sec. 3.2):
//   encode(call 1) -> combine -> encode(call 2) -> combine -> decode(call 3).
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <string.h>

#include "flarepp_internal.h"

namespace flarepp {
namespace {

constexpr int64_t kMaxM = 2048;
constexpr int64_t kMaxTokenHeads = int64_t(1) << 40;  // B*H*N limit (index headroom)
constexpr size_t kWsAlign = 256;
constexpr int kStageEvents = 6;
constexpr int64_t kMaxTmaCoord = 2147483647 - 4096;  // TMA coordinates are signed 32-bit
constexpr int64_t kTcItem = 64;               // tokens per tensor-core encode item

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

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
        // waves x (64-token items per unit, scaled by the group's route tiles, + a fixed
        // per-unit cost of about three items).
        p->tc_group = tc_group_rows(s->D);
        p->n_groups = cdiv(s->M, p->tc_group);
        p->sub_per_chunk = 4;
        const int64_t ns = p->tc_group / 128;
        const int64_t tiles0 = s->M >= p->tc_group ? ns : cdiv(s->M, 128);
        const double na = tiles0 <= 1 ? 1.0 : (tiles0 <= 2 ? 2.0 : 4.0);
        const int64_t per_chunk = bh * p->n_groups;
        const int64_t max_chunks = cdiv(s->N, kTcItem);
        double best = 1e300;
        int64_t best_n = 1;
        for (int64_t n = 1; n <= max_chunks && n <= 65536; ++n) {
            const int64_t waves = cdiv(per_chunk * n, kNumSMs);
            const int64_t items = cdiv(cdiv(s->N, n), kTcItem);
            const double cost = (double)waves * ((double)items * na / (double)ns + 3.0);
            if (cost < best) {
                best = cost;
                best_n = n;
            }
        }
        p->chunk_len = cdiv(cdiv(s->N, best_n), kTcItem) * kTcItem;
        p->nchunk = cdiv(s->N, p->chunk_len);
    }

    const size_t rows =
        (size_t)bh * (size_t)p->nchunk * (size_t)p->sub_per_chunk * (size_t)s->M;
    size_t off = 0;
    p->off_status = off;
    off = align_up(off + sizeof(int32_t), kWsAlign);
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
        p->off_seedneg = off;
        off = align_up(off + (size_t)s->H * (size_t)s->M * (size_t)s->D * 2, kWsAlign);
    }
    p->total = off;
    return FLAREPP_OK;
}

namespace {

bool aligned16(const void* ptr) { return ((uintptr_t)ptr & 15u) == 0; }

bool overlaps(const void* a, size_t na, const void* b, size_t nb) {
    if (!a || !b || na == 0 || nb == 0) return false;
    const uintptr_t a0 = (uintptr_t)a, b0 = (uintptr_t)b;
    return a0 < b0 + nb && b0 < a0 + na;
}

flarepp_status route_impl(const flarepp_shape* shape, const void* seeds, const void* Kt,
                          const void* Vt, const void* K, const void* V, float scale, void* Y,
                          void* workspace, size_t workspace_bytes, void* stream, float* Q_out,
                          float* Z_out, void* const* events, int n_events) {
    Plan p;
    flarepp_status stt = make_plan(shape, &p);
    if (stt != FLAREPP_OK) return stt;
    if (!isfinite(scale)) return FLAREPP_ERR_INVALID_ARGUMENT;
    cudaStream_t st = (cudaStream_t)stream;
    const size_t elt = p.dtype == FLAREPP_F32 ? 4 : 2;
    const size_t tok_bytes = (size_t)p.BH * (size_t)p.N * (size_t)p.D * elt;
    const size_t seed_bytes = (size_t)p.H * (size_t)p.M * (size_t)p.D * elt;
    const size_t qz_bytes = (size_t)p.BH * (size_t)p.M * (size_t)p.D * sizeof(float);

    // pointer checks (only buffers with a non-zero size must exist)
    if (tok_bytes) {
        const void* ptrs[5] = {Kt, Vt, K, V, Y};
        for (const void* q : ptrs)
            if (!q || !aligned16(q)) return FLAREPP_ERR_INVALID_ARGUMENT;
        const void* ins[4] = {Kt, Vt, K, V};
        for (const void* q : ins)
            if (overlaps(Y, tok_bytes, q, tok_bytes)) return FLAREPP_ERR_INVALID_ARGUMENT;
        if (overlaps(Y, tok_bytes, seeds, seed_bytes)) return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    if (seed_bytes && tok_bytes && (!seeds || !aligned16(seeds)))
        return FLAREPP_ERR_INVALID_ARGUMENT;
    if (events) {
        if (n_events < kStageEvents) return FLAREPP_ERR_INVALID_ARGUMENT;
        for (int i = 0; i < kStageEvents; ++i)
            if (!events[i]) return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    if (qz_bytes) {
        if ((Q_out && !aligned16(Q_out)) || (Z_out && !aligned16(Z_out)))
            return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    if (p.total) {
        if (!workspace || ((uintptr_t)workspace % kWsAlign) != 0) return FLAREPP_ERR_WORKSPACE;
        if (workspace_bytes < p.total) return FLAREPP_ERR_WORKSPACE;
        if (overlaps(Y, tok_bytes, workspace, p.total)) return FLAREPP_ERR_INVALID_ARGUMENT;
    }

    // degenerate shapes
    if (p.BH == 0) return FLAREPP_OK;
    if (p.N == 0) {  // every encoder row has no keys: Q = Z = 0 (App. A.3); Y is empty
        if (Q_out && qz_bytes && cudaMemsetAsync(Q_out, 0, qz_bytes, st) != cudaSuccess)
            return FLAREPP_ERR_CUDA;
        if (Z_out && qz_bytes && cudaMemsetAsync(Z_out, 0, qz_bytes, st) != cudaSuccess)
            return FLAREPP_ERR_CUDA;
        return FLAREPP_OK;
    }
    if (p.M == 0) {  // every decode row has no keys: Y = 0
        return cudaMemsetAsync(Y, 0, tok_bytes, st) == cudaSuccess ? FLAREPP_OK : FLAREPP_ERR_CUDA;
    }

    char* ws = (char*)workspace;
    const bool tc = p.path == kPathTc;
    const bool neg = scale < 0.f;
    auto mark = [&](int i) {
        return !events || cudaEventRecord((cudaEvent_t)events[i], st) == cudaSuccess;
    };
    auto encode = [&](int call, const void* k, const void* v) {
        return tc ? tc_encode(p, call, k, v, seeds, scale, ws, st)
                  : simt_encode_f32(p, call, k, v, seeds, scale, ws, st);
    };
    if (cudaMemsetAsync(ws + p.off_status, 0, sizeof(int32_t), st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    if (tc && neg &&
        negate_bf16(seeds, ws + p.off_seedneg, p.H * p.M * p.D, st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    if (!mark(0)) return FLAREPP_ERR_CUDA;
    if (encode(1, Kt, Vt) != cudaSuccess || !mark(1)) return FLAREPP_ERR_CUDA;
    if (combine(p, 1, ws, neg, st) != cudaSuccess || !mark(2)) return FLAREPP_ERR_CUDA;
    if (encode(2, K, V) != cudaSuccess || !mark(3)) return FLAREPP_ERR_CUDA;
    if (combine(p, 2, ws, false, st) != cudaSuccess || !mark(4)) return FLAREPP_ERR_CUDA;
    cudaError_t e;
    e = tc ? tc_decode(p, K, scale, Y, ws, st) : simt_decode_f32(p, K, scale, Y, ws, st);
    if (e != cudaSuccess || !mark(5)) return FLAREPP_ERR_CUDA;
    if (Q_out && cudaMemcpyAsync(Q_out, ws + p.off_q32, qz_bytes, cudaMemcpyDeviceToDevice, st) !=
                     cudaSuccess)
        return FLAREPP_ERR_CUDA;
    if (Z_out && cudaMemcpyAsync(Z_out, ws + p.off_z32, qz_bytes, cudaMemcpyDeviceToDevice, st) !=
                     cudaSuccess)
        return FLAREPP_ERR_CUDA;
    return FLAREPP_OK;
}

}  // namespace
}  // namespace flarepp

extern "C" {

size_t flarepp_route_workspace_bytes(const flarepp_shape* shape) {
    flarepp::Plan p;
    if (flarepp::make_plan(shape, &p) != FLAREPP_OK) return 0;
    return p.total;
}

flarepp_status flarepp_route_fwd(const flarepp_shape* shape, const void* seeds, const void* Kt,
                                 const void* Vt, const void* K, const void* V, float scale,
                                 void* Y, void* workspace, size_t workspace_bytes, void* stream) {
    return flarepp::route_impl(shape, seeds, Kt, Vt, K, V, scale, Y, workspace, workspace_bytes,
                               stream, nullptr, nullptr, nullptr, 0);
}

flarepp_status flarepp_route_fwd_debug(const flarepp_shape* shape, const void* seeds,
                                       const void* Kt, const void* Vt, const void* K,
                                       const void* V, float scale, void* Y, void* workspace,
                                       size_t workspace_bytes, void* stream, float* Q_out,
                                       float* Z_out) {
    return flarepp::route_impl(shape, seeds, Kt, Vt, K, V, scale, Y, workspace, workspace_bytes,
                               stream, Q_out, Z_out, nullptr, 0);
}

flarepp_status flarepp_route_fwd_profiled(const flarepp_shape* shape, const void* seeds,
                                          const void* Kt, const void* Vt, const void* K,
                                          const void* V, float scale, void* Y, void* workspace,
                                          size_t workspace_bytes, void* stream,
                                          void* const* events, int n_events) {
    if (!events) return FLAREPP_ERR_INVALID_ARGUMENT;
    return flarepp::route_impl(shape, seeds, Kt, Vt, K, V, scale, Y, workspace, workspace_bytes,
                               stream, nullptr, nullptr, events, n_events);
}

flarepp_status flarepp_route_device_status(const flarepp_shape* shape, const void* workspace,
                                          void* stream, int32_t* status_out) {
    flarepp::Plan p;
    if (!status_out) return FLAREPP_ERR_INVALID_ARGUMENT;
    const flarepp_status s = flarepp::make_plan(shape, &p);
    if (s != FLAREPP_OK) return s;
    *status_out = FLAREPP_OK;
    if (p.total == 0) return FLAREPP_OK;
    if (!workspace) return FLAREPP_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    if (cudaMemcpyAsync(status_out, (const char*)workspace + p.off_status, sizeof(int32_t),
                        cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    return FLAREPP_OK;
}

const char* flarepp_status_string(flarepp_status status) {
    switch (status) {
        case FLAREPP_OK: return "ok";
        case FLAREPP_ERR_INVALID_ARGUMENT: return "invalid argument";
        case FLAREPP_ERR_UNSUPPORTED: return "unsupported shape";
        case FLAREPP_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
        case FLAREPP_ERR_CUDA: return "CUDA launch or call failed";
        case FLAREPP_ERR_TIMEOUT: return "bounded device wait timed out";
    }
    return "unknown status";
}

const char* flarepp_version(void) { return "0.1.0"; }

}  // extern "C"
