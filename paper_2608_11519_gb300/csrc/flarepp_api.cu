// The C ABI of libflarepp: argument checks and the launch sequence of the routing chain
// (Sec. 3.2):
//   encode(call 1) -> combine -> encode(call 2) -> combine -> decode(call 3).
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <string.h>

#include <mutex>
#include <utility>
#include <vector>

#include "flarepp_internal.h"

namespace flarepp {

cudaError_t ensure_smem_limit(const void* func, int bytes) {
    constexpr int kMaxDevices = 64;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    static std::mutex mu;
    static std::vector<std::pair<const void*, uint64_t>> done;  // kernel, devices set
    std::lock_guard<std::mutex> lock(mu);
    for (auto& d : done)
        if (d.first == func) {
            if (d.second >> dev & 1u) return cudaSuccess;
            e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
            if (e == cudaSuccess) d.second |= uint64_t(1) << dev;
            return e;
        }
    e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) done.emplace_back(func, uint64_t(1) << dev);
    return e;
}

namespace {

constexpr int kStageEvents = 6;

bool aligned16(const void* ptr) { return ((uintptr_t)ptr & 15u) == 0; }

bool overlaps(const void* a, size_t na, const void* b, size_t nb) {
    if (!a || !b || na == 0 || nb == 0) return false;
    const uintptr_t a0 = (uintptr_t)a, b0 = (uintptr_t)b;
    return a0 < b0 + nb && b0 < a0 + na;
}

bool spans_overlap(const void* const* ptrs, const size_t* bytes, int n, const void* p,
                   size_t nb) {
    for (int i = 0; i < n; ++i)
        if (overlaps(p, nb, ptrs[i], bytes[i])) return true;
    return false;
}

flarepp_status route_impl(const flarepp_shape* shape, const void* seeds, const void* Kt,
                          const void* Vt, const void* K, const void* V, float scale, void* Y,
                          void* workspace, size_t workspace_bytes, void* stream, float* Q_out,
                          float* Z_out, void* const* events, int n_events,
                          bool reset_status = true, char* saved = nullptr) {
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
        // the kernels write the workspace while they read the inputs
        const void* ins[5] = {seeds, Kt, Vt, K, V};
        const size_t nb[5] = {seed_bytes, tok_bytes, tok_bytes, tok_bytes, tok_bytes};
        if (spans_overlap(ins, nb, 5, workspace, p.total)) return FLAREPP_ERR_INVALID_ARGUMENT;
        float* const qz[2] = {Q_out, Z_out};
        for (float* q : qz)
            if (q && qz_bytes &&
                (overlaps(q, qz_bytes, workspace, p.total) || overlaps(q, qz_bytes, Y, tok_bytes)))
                return FLAREPP_ERR_INVALID_ARGUMENT;
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
    // The training forward (D <= 32) gives the scores of calls 2 and 3 Q as a hi/lo pair of
    // bf16 operands, so that the function its backward differentiates sees Q to about 2^-17
    // (with bf16 Q alone, sharp softmaxes move the gradient by several percent).
    const bool lo = tc && saved && p.D <= 32;
    auto encode = [&](int call, const void* k, const void* v) {
        return tc ? tc_encode(p, call, k, v, seeds, scale, ws, st, lo)
                  : simt_encode_f32(p, call, k, v, seeds, scale, ws, st);
    };
    if (reset_status && cudaMemsetAsync(ws + p.off_status, 0, sizeof(int32_t), st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    if (tc && cudaMemsetAsync(ws + p.off_overflow, 0, 3 * sizeof(int32_t), st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    if (tc && neg &&
        negate_bf16(seeds, ws + p.off_seedneg, p.H * p.M * p.D, st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    if (!mark(0)) return FLAREPP_ERR_CUDA;
    if (encode(1, Kt, Vt) != cudaSuccess || !mark(1)) return FLAREPP_ERR_CUDA;
    // the training forward keeps each call's log-normaliser for the backward (App. A.5)
    const SavedLayout sv = saved_layout(p);
    float* l1 = saved ? (float*)(saved + sv.off_l1) : nullptr;
    float* l2 = saved ? (float*)(saved + sv.off_l2) : nullptr;
    float* l3 = saved ? (float*)(saved + sv.off_l3) : nullptr;
    if (combine(p, 1, ws, neg, st, l1, lo) != cudaSuccess || !mark(2)) return FLAREPP_ERR_CUDA;
    if (encode(2, K, V) != cudaSuccess || !mark(3)) return FLAREPP_ERR_CUDA;
    if (combine(p, 2, ws, false, st, l2) != cudaSuccess || !mark(4)) return FLAREPP_ERR_CUDA;
    cudaError_t e;
    e = tc ? tc_decode(p, K, scale, Y, ws, st, l3, lo)
           : simt_decode_f32(p, K, scale, Y, ws, st, l3);
    if (e != cudaSuccess || !mark(5)) return FLAREPP_ERR_CUDA;
    if (saved) {
        Q_out = (float*)(saved + sv.off_q);
        Z_out = (float*)(saved + sv.off_z);
    }
    if (Q_out && cudaMemcpyAsync(Q_out, ws + p.off_q32, qz_bytes, cudaMemcpyDeviceToDevice, st) !=
                     cudaSuccess)
        return FLAREPP_ERR_CUDA;
    if (Z_out && cudaMemcpyAsync(Z_out, ws + p.off_z32, qz_bytes, cudaMemcpyDeviceToDevice, st) !=
                     cudaSuccess)
        return FLAREPP_ERR_CUDA;
    return FLAREPP_OK;
}

// ---------------------------------------------------------------- FLARE (fixed queries)

// FLARE (Sec. 3, eq. prelim_flare_sdpa): Z = SDPA(Q_h, K, V), Y = SDPA(K, Q_h, Z) with learned
// queries Q [H, M, D] shared by the batch. The routing chain without its first call: the
// encode runs as call 1 does (A = the per-head queries), its merge writes Z, and the decode
// reads a per-(b, h) copy of Q as its keys.
flarepp_status flare_impl(const flarepp_shape* shape, const void* Qh, const void* K, const void* V,
                          float scale, void* Y, void* workspace, size_t workspace_bytes,
                          void* stream, float* Z_out, bool reset_status = true) {
    Plan p;
    flarepp_status stt = make_plan(shape, &p);
    if (stt != FLAREPP_OK) return stt;
    if (!isfinite(scale)) return FLAREPP_ERR_INVALID_ARGUMENT;
    cudaStream_t st = (cudaStream_t)stream;
    const size_t elt = p.dtype == FLAREPP_F32 ? 4 : 2;
    const size_t tok_bytes = (size_t)p.BH * (size_t)p.N * (size_t)p.D * elt;
    const size_t q_bytes = (size_t)p.H * (size_t)p.M * (size_t)p.D * elt;
    const size_t z_bytes = (size_t)p.BH * (size_t)p.M * (size_t)p.D * sizeof(float);
    if (tok_bytes) {
        const void* ptrs[3] = {K, V, Y};
        for (const void* q : ptrs)
            if (!q || !aligned16(q)) return FLAREPP_ERR_INVALID_ARGUMENT;
        if (overlaps(Y, tok_bytes, K, tok_bytes) || overlaps(Y, tok_bytes, V, tok_bytes) ||
            overlaps(Y, tok_bytes, Qh, q_bytes))
            return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    if (q_bytes && tok_bytes && (!Qh || !aligned16(Qh))) return FLAREPP_ERR_INVALID_ARGUMENT;
    if (z_bytes && Z_out && !aligned16(Z_out)) return FLAREPP_ERR_INVALID_ARGUMENT;
    if (p.total) {
        if (!workspace || ((uintptr_t)workspace % kWsAlign) != 0) return FLAREPP_ERR_WORKSPACE;
        if (workspace_bytes < p.total) return FLAREPP_ERR_WORKSPACE;
        if (overlaps(Y, tok_bytes, workspace, p.total)) return FLAREPP_ERR_INVALID_ARGUMENT;
        const void* ins[3] = {Qh, K, V};
        const size_t nb[3] = {q_bytes, tok_bytes, tok_bytes};
        if (spans_overlap(ins, nb, 3, workspace, p.total)) return FLAREPP_ERR_INVALID_ARGUMENT;
        if (Z_out && z_bytes &&
            (overlaps(Z_out, z_bytes, workspace, p.total) || overlaps(Z_out, z_bytes, Y, tok_bytes)))
            return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    if (p.BH == 0) return FLAREPP_OK;
    if (p.N == 0) {  // every route has no keys: Z = 0 (App. A.3); Y is empty
        if (Z_out && z_bytes && cudaMemsetAsync(Z_out, 0, z_bytes, st) != cudaSuccess)
            return FLAREPP_ERR_CUDA;
        return FLAREPP_OK;
    }
    if (p.M == 0)
        return cudaMemsetAsync(Y, 0, tok_bytes, st) == cudaSuccess ? FLAREPP_OK : FLAREPP_ERR_CUDA;

    char* ws = (char*)workspace;
    const bool tc = p.path == kPathTc;
    const bool neg = scale < 0.f;
    if (reset_status && cudaMemsetAsync(ws + p.off_status, 0, sizeof(int32_t), st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    if (tc && cudaMemsetAsync(ws + p.off_overflow, 0, 3 * sizeof(int32_t), st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    // the encode of call 1 with the learned queries, merged into Z
    if (tc && neg && negate_bf16(Qh, ws + p.off_seedneg, p.H * p.M * p.D, st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    cudaError_t e = tc ? tc_encode(p, 1, K, V, Qh, scale, ws, st)
                       : simt_encode_f32(p, 1, K, V, Qh, scale, ws, st);
    if (e != cudaSuccess || combine(p, 2, ws, false, st) != cudaSuccess) return FLAREPP_ERR_CUDA;
    // the decode's keys: Q for every batch element (on the tensor-core path the bf16 operand,
    // negated for a negative scale as the chain's call-1 merge does)
    const void* qsrc = tc && neg ? (const void*)(ws + p.off_seedneg) : Qh;
    char* qdst = ws + (tc ? p.off_qop : p.off_q32);
    for (int64_t b = 0; b < p.B; ++b)
        if (cudaMemcpyAsync(qdst + (size_t)b * q_bytes, qsrc, q_bytes, cudaMemcpyDeviceToDevice,
                            st) != cudaSuccess)
            return FLAREPP_ERR_CUDA;
    e = tc ? tc_decode(p, K, scale, Y, ws, st) : simt_decode_f32(p, K, scale, Y, ws, st);
    if (e != cudaSuccess) return FLAREPP_ERR_CUDA;
    if (Z_out && cudaMemcpyAsync(Z_out, ws + p.off_z32, z_bytes, cudaMemcpyDeviceToDevice, st) !=
                     cudaSuccess)
        return FLAREPP_ERR_CUDA;
    return FLAREPP_OK;
}

// ---------------------------------------------------------------- the chain on host buffers

// Heads of one pipeline group: a run of consecutive (b, h) slices, either a block of heads
// of one batch element or whole batch elements (so that every group is a valid shape).
struct HostGroups {
    int64_t len;  // (b, h) slices per group
    int64_t n;    // groups
};

HostGroups host_groups(const Plan& p) {
    constexpr int64_t kTarget = 8;  // measured best for mesh3d (8 heads): 12.0 ms vs 12.5 (4)
    const int64_t bh = p.BH;
    int64_t want = (bh + kTarget - 1) / kTarget;
    if (want < 1) want = 1;
    int64_t len;
    if (want >= p.H) {
        len = (want + p.H - 1) / p.H * p.H;  // whole batch elements
    } else {
        len = p.H;  // the smallest divisor of H that is at least `want`
        for (int64_t d = want; d <= p.H; ++d)
            if (p.H % d == 0) {
                len = d;
                break;
            }
    }
    if (len > bh) len = bh;
    HostGroups g;
    g.len = len;
    g.n = (bh + len - 1) / len;
    return g;
}

// Layout of the device buffer of flarepp_route_fwd_host: the workspace of one group first
// (so that its status word sits at offset 0), then the device copies of the inputs and Y.
struct HostLayout {
    flarepp_shape group;  // shape of a full group
    size_t ws_bytes;
    size_t off_seeds, off_kt, off_vt, off_k, off_v, off_y, total;
};

bool host_layout(const flarepp_shape* s, const Plan& p, const HostGroups& g, HostLayout* L) {
    const size_t elt = p.dtype == FLAREPP_F32 ? 4 : 2;
    const size_t tok = (size_t)p.BH * (size_t)p.N * (size_t)p.D * elt;
    const size_t seed = (size_t)p.H * (size_t)p.M * (size_t)p.D * elt;
    L->group = *s;
    if (g.len >= p.H) {
        L->group.B = g.len / p.H;
    } else {
        L->group.B = 1;
        L->group.H = g.len;
    }
    Plan gp;
    if (make_plan(&L->group, &gp) != FLAREPP_OK) return false;
    L->ws_bytes = gp.total;
    const int64_t last = p.BH - (g.n - 1) * g.len;  // a shorter last group of batch elements
    if (last != g.len) {
        flarepp_shape ls = L->group;
        ls.B = last / p.H;
        if (make_plan(&ls, &gp) != FLAREPP_OK) return false;
        if (gp.total > L->ws_bytes) L->ws_bytes = gp.total;
    }
    size_t off = align_up(L->ws_bytes, kWsAlign);
    L->off_seeds = off;
    off = align_up(off + seed, kWsAlign);
    L->off_kt = off;
    off = align_up(off + tok, kWsAlign);
    L->off_vt = off;
    off = align_up(off + tok, kWsAlign);
    L->off_k = off;
    off = align_up(off + tok, kWsAlign);
    L->off_v = off;
    off = align_up(off + tok, kWsAlign);
    L->off_y = off;
    off = align_up(off + tok, kWsAlign);
    L->total = off;
    return true;
}

// The chain (or, with `flare`, FLARE with the learned queries in seeds_h, K~ = K and V~ = V)
// on host buffers.
flarepp_status route_host_impl(const flarepp_shape* shape, const void* seeds_h, const void* Kt_h,
                               const void* Vt_h, const void* K_h, const void* V_h, float scale,
                               void* Y_h, void* dbuf, size_t dbuf_bytes, void* stream,
                               bool flare = false) {
    Plan p;
    flarepp_status stt = make_plan(shape, &p);
    if (stt != FLAREPP_OK) return stt;
    if (!isfinite(scale)) return FLAREPP_ERR_INVALID_ARGUMENT;
    if (p.BH == 0 || p.N == 0) return FLAREPP_OK;  // Y is empty
    const size_t elt = p.dtype == FLAREPP_F32 ? 4 : 2;
    const size_t tok = (size_t)p.BH * (size_t)p.N * (size_t)p.D * elt;
    const size_t seed = (size_t)p.H * (size_t)p.M * (size_t)p.D * elt;
    {
        const void* ptrs[5] = {Kt_h, Vt_h, K_h, V_h, Y_h};
        for (const void* q : ptrs)
            if (!q) return FLAREPP_ERR_INVALID_ARGUMENT;
        const void* ins[4] = {Kt_h, Vt_h, K_h, V_h};
        for (const void* q : ins)
            if (overlaps(Y_h, tok, q, tok)) return FLAREPP_ERR_INVALID_ARGUMENT;
        if (seed && (!seeds_h || overlaps(Y_h, tok, seeds_h, seed)))
            return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    const HostGroups g = host_groups(p);
    HostLayout L;
    if (!host_layout(shape, p, g, &L)) return FLAREPP_ERR_UNSUPPORTED;
    if (!dbuf || ((uintptr_t)dbuf % kWsAlign) != 0 || dbuf_bytes < L.total)
        return FLAREPP_ERR_WORKSPACE;
    char* db = (char*)dbuf;
    cudaStream_t st = (cudaStream_t)stream;

    // two streams of the library's own (inputs in, Y out) and the events that order them
    // against `stream`; each is released when its work is done
    constexpr int kMaxEvents = 2 * 64 + 2;
    cudaStream_t cin = nullptr, cout = nullptr;
    cudaEvent_t ev[kMaxEvents] = {};
    int n_ev = 0;
    if (g.n > 64) return FLAREPP_ERR_UNSUPPORTED;  // not reached: host_groups makes at most 8
    flarepp_status rc = FLAREPP_OK;
    auto cleanup = [&]() {
        for (int i = 0; i < n_ev; ++i) cudaEventDestroy(ev[i]);
        if (cin) cudaStreamDestroy(cin);
        if (cout) cudaStreamDestroy(cout);
    };
    auto new_event = [&](cudaEvent_t* e) {
        if (cudaEventCreateWithFlags(e, cudaEventDisableTiming) != cudaSuccess) return false;
        ev[n_ev++] = *e;
        return true;
    };
    cudaEvent_t e_start, e_end;
    if (cudaStreamCreateWithFlags(&cin, cudaStreamNonBlocking) != cudaSuccess ||
        cudaStreamCreateWithFlags(&cout, cudaStreamNonBlocking) != cudaSuccess ||
        !new_event(&e_start) || !new_event(&e_end)) {
        cleanup();
        return FLAREPP_ERR_CUDA;
    }
    const size_t gtok = (size_t)g.len * (size_t)p.N * (size_t)p.D * elt;  // bytes of a group
    bool ok = cudaEventRecord(e_start, st) == cudaSuccess &&
              cudaStreamWaitEvent(cin, e_start, 0) == cudaSuccess &&
              cudaStreamWaitEvent(cout, e_start, 0) == cudaSuccess;
    if (ok && seed)
        ok = cudaMemcpyAsync(db + L.off_seeds, seeds_h, seed, cudaMemcpyHostToDevice, cin) ==
             cudaSuccess;
    // inputs of every group, in order, on the input stream. With the shared projection
    // (Kt = K and Vt = V on the host, App. cost_model) K and V are copied once and serve as
    // both pairs.
    const bool shared = Kt_h == K_h && Vt_h == V_h;
    const size_t off_kt = shared ? L.off_k : L.off_kt, off_vt = shared ? L.off_v : L.off_vt;
    cudaEvent_t e_in[64], e_done[64];
    for (int64_t k = 0; ok && k < g.n; ++k) {
        const size_t o = (size_t)k * gtok;
        const size_t n = o + gtok <= tok ? gtok : tok - o;
        const void* src[4] = {K_h, V_h, Kt_h, Vt_h};
        const size_t dst[4] = {L.off_k, L.off_v, L.off_kt, L.off_vt};
        for (int t = 0; ok && t < (shared ? 2 : 4); ++t)
            ok = cudaMemcpyAsync(db + dst[t] + o, (const char*)src[t] + o, n,
                                 cudaMemcpyHostToDevice, cin) == cudaSuccess;
        ok = ok && new_event(&e_in[k]) && new_event(&e_done[k]) &&
             cudaEventRecord(e_in[k], cin) == cudaSuccess;
    }
    // the chain of each group on `stream`, and its Y back on the output stream
    for (int64_t k = 0; ok && k < g.n; ++k) {
        const int64_t bh0 = k * g.len;
        const int64_t len = bh0 + g.len <= p.BH ? g.len : p.BH - bh0;
        flarepp_shape gs = L.group;
        if (len >= p.H) gs.B = len / p.H;  // a shorter last group of whole batch elements
        const size_t o = (size_t)bh0 * (size_t)p.N * (size_t)p.D * elt;
        const size_t n = (size_t)len * (size_t)p.N * (size_t)p.D * elt;
        const size_t so = (size_t)(bh0 % p.H) * (size_t)p.M * (size_t)p.D * elt;
        ok = cudaStreamWaitEvent(st, e_in[k], 0) == cudaSuccess;
        if (!ok) break;
        rc = flare ? flare_impl(&gs, db + L.off_seeds + so, db + L.off_k + o, db + L.off_v + o,
                                scale, db + L.off_y + o, db, L.ws_bytes, st, nullptr, k == 0)
                   : route_impl(&gs, db + L.off_seeds + so, db + off_kt + o, db + off_vt + o,
                                db + L.off_k + o, db + L.off_v + o, scale, db + L.off_y + o, db,
                                L.ws_bytes, st, nullptr, nullptr, nullptr, 0, k == 0);
        if (rc != FLAREPP_OK) break;
        ok = cudaEventRecord(e_done[k], st) == cudaSuccess &&
             cudaStreamWaitEvent(cout, e_done[k], 0) == cudaSuccess &&
             cudaMemcpyAsync((char*)Y_h + o, db + L.off_y + o, n, cudaMemcpyDeviceToHost, cout) ==
                 cudaSuccess;
    }
    // later work on `stream` follows the last copy of Y
    if (ok && rc == FLAREPP_OK)
        ok = cudaEventRecord(e_end, cout) == cudaSuccess &&
             cudaStreamWaitEvent(st, e_end, 0) == cudaSuccess;
    cleanup();
    if (rc != FLAREPP_OK) return rc;
    return ok ? FLAREPP_OK : FLAREPP_ERR_CUDA;
}

// ---------------------------------------------------------------- training forward, backward

flarepp_status route_fwd_train_impl(const flarepp_shape* shape, const void* seeds, const void* Kt,
                                    const void* Vt, const void* K, const void* V, float scale,
                                    void* Y, void* saved, size_t saved_bytes, void* workspace,
                                    size_t workspace_bytes, void* stream) {
    Plan p;
    flarepp_status stt = make_plan(shape, &p);
    if (stt != FLAREPP_OK) return stt;
    const SavedLayout sv = saved_layout(p);
    if (p.BH && p.N && p.M) {
        if (!saved || !aligned16(saved) || saved_bytes < sv.total)
            return FLAREPP_ERR_INVALID_ARGUMENT;
        const size_t elt = p.dtype == FLAREPP_F32 ? 4 : 2;
        const size_t tok_bytes = (size_t)p.BH * (size_t)p.N * (size_t)p.D * elt;
        const void* ins[6] = {Kt, Vt, K, V, Y, workspace};
        const size_t nb[6] = {tok_bytes, tok_bytes, tok_bytes, tok_bytes, tok_bytes, p.total};
        if (spans_overlap(ins, nb, 6, saved, sv.total)) return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    return route_impl(shape, seeds, Kt, Vt, K, V, scale, Y, workspace, workspace_bytes, stream,
                      nullptr, nullptr, nullptr, 0, true, (char*)saved);
}

flarepp_status route_bwd_impl(const flarepp_shape* shape, const void* seeds, const void* Kt,
                              const void* Vt, const void* K, const void* V, float scale,
                              const void* Y, const void* dY, const void* saved,
                              size_t saved_bytes, void* dseeds, void* dKt, void* dVt, void* dK,
                              void* dV, void* workspace, size_t workspace_bytes, void* stream) {
    Plan p;
    flarepp_status stt = make_plan(shape, &p);
    if (stt != FLAREPP_OK) return stt;
    if (!isfinite(scale)) return FLAREPP_ERR_INVALID_ARGUMENT;
    cudaStream_t st = (cudaStream_t)stream;
    const BwdPlan bp = make_bwd_plan(p);
    const SavedLayout sv = saved_layout(p);
    const size_t elt = p.dtype == FLAREPP_F32 ? 4 : 2;
    const size_t tok = (size_t)p.BH * (size_t)p.N * (size_t)p.D * elt;
    const size_t seed = (size_t)p.H * (size_t)p.M * (size_t)p.D * elt;
    const bool work = p.BH && p.N && p.M;
    // outputs: present and aligned where non-empty, disjoint from every input and each other
    void* outs[5] = {dseeds, dKt, dVt, dK, dV};
    const size_t ob[5] = {seed, tok, tok, tok, tok};
    for (int i = 0; i < 5; ++i)
        if (ob[i] && (!outs[i] || !aligned16(outs[i]))) return FLAREPP_ERR_INVALID_ARGUMENT;
    if (work) {
        const void* ins[9] = {seeds, Kt, Vt, K, V, Y, dY, saved, workspace};
        const size_t ib[9] = {seed, tok, tok, tok, tok, tok, tok, sv.total, bp.total};
        for (int i = 0; i < 7; ++i)
            if (!ins[i] || !aligned16(ins[i])) return FLAREPP_ERR_INVALID_ARGUMENT;
        if (!saved || !aligned16(saved) || saved_bytes < sv.total)
            return FLAREPP_ERR_INVALID_ARGUMENT;
        if (!workspace || ((uintptr_t)workspace % kWsAlign) != 0 || workspace_bytes < bp.total)
            return FLAREPP_ERR_WORKSPACE;
        for (int i = 0; i < 5; ++i) {
            if (spans_overlap(ins, ib, 9, outs[i], ob[i])) return FLAREPP_ERR_INVALID_ARGUMENT;
            for (int j = 0; j < i; ++j)
                if (overlaps(outs[i], ob[i], outs[j], ob[j])) return FLAREPP_ERR_INVALID_ARGUMENT;
        }
        if (spans_overlap(ins, ib, 8, workspace, bp.total)) return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    // degenerate shapes: every gradient that exists is zero
    if (!work) {
        for (int i = 0; i < 5; ++i)
            if (ob[i] && cudaMemsetAsync(outs[i], 0, ob[i], st) != cudaSuccess)
                return FLAREPP_ERR_CUDA;
        return FLAREPP_OK;
    }
    char* ws = (char*)workspace;
    if (cudaMemsetAsync(ws + bp.off_status, 0, sizeof(int32_t), st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    const cudaError_t e = route_bwd(p, bp, seeds, Kt, Vt, K, V, scale, Y, dY,
                                    (const char*)saved, dseeds, dKt, dVt, dK, dV, ws, st);
    return e == cudaSuccess ? FLAREPP_OK : FLAREPP_ERR_CUDA;
}

// ---------------------------------------------------------------- the mixer layer

// Workspace of flarepp_mixer_fwd: the chain's workspace first (its status word at offset 0),
// then the projections (K, V and, for four projections, K~, V~) and Y, each [B][H][N][D] bf16.
struct MixerLayout {
    size_t off_proj[4], off_y, total;
};

bool mixer_layout(const Plan& p, int n_proj, MixerLayout* L) {
    const size_t tok = (size_t)p.BH * (size_t)p.N * (size_t)p.D * 2;
    size_t off = align_up(p.total, kWsAlign);
    for (int i = 0; i < 4; ++i) {
        L->off_proj[i] = off;
        if (i < n_proj) off = align_up(off + tok, kWsAlign);
    }
    L->off_y = off;
    off = align_up(off + tok, kWsAlign);
    L->total = off;
    return true;
}

// State a training forward of the mixer keeps for its backward: the chain's saved state,
// then Y and the n_proj projections (K, V, K~, V~), each [B][H][N][D] bf16. The forward
// writes the projections there directly, so keeping them costs memory only, and the
// backward does not recompute them.
struct MixerSaved {
    size_t off_y, off_proj[4], total;
};

MixerSaved mixer_saved(const Plan& p, int n_proj) {
    const size_t tok = (size_t)p.BH * (size_t)p.N * (size_t)p.D * 2;
    MixerSaved m;
    size_t off = align_up(saved_layout(p).total, kWsAlign);
    m.off_y = off;
    off = align_up(off + tok, kWsAlign);
    for (int i = 0; i < 4; ++i) {
        m.off_proj[i] = off;
        if (i < n_proj) off = align_up(off + tok, kWsAlign);
    }
    m.total = off;
    return m;
}

flarepp_status mixer_impl(const flarepp_shape* shape, int n_proj, const void* X, const void* W_in,
                          const void* Wo, const void* seeds, float scale, void* O,
                          void* workspace, size_t workspace_bytes, void* stream,
                          void* const* events = nullptr, char* saved = nullptr) {
    Plan p;
    flarepp_status stt = make_plan(shape, &p);
    if (stt != FLAREPP_OK) return stt;
    if (n_proj != 2 && n_proj != 4) return FLAREPP_ERR_INVALID_ARGUMENT;
    if (p.dtype != FLAREPP_BF16) return FLAREPP_ERR_UNSUPPORTED;  // tensor-core GEMMs only
    if (!isfinite(scale)) return FLAREPP_ERR_INVALID_ARGUMENT;
    cudaStream_t st = (cudaStream_t)stream;
    const int64_t C = p.H * p.D;
    const size_t x_bytes = (size_t)p.B * (size_t)p.N * (size_t)C * 2;
    const size_t w_bytes = (size_t)n_proj * (size_t)C * (size_t)C * 2;
    const size_t wo_bytes = (size_t)C * (size_t)C * 2;
    const size_t seed_bytes = (size_t)p.H * (size_t)p.M * (size_t)p.D * 2;
    if (x_bytes) {
        const void* ptrs[4] = {X, W_in, Wo, O};
        for (const void* q : ptrs)
            if (!q || !aligned16(q)) return FLAREPP_ERR_INVALID_ARGUMENT;
        if (overlaps(O, x_bytes, X, x_bytes) || overlaps(O, x_bytes, W_in, w_bytes) ||
            overlaps(O, x_bytes, Wo, wo_bytes) || overlaps(O, x_bytes, seeds, seed_bytes))
            return FLAREPP_ERR_INVALID_ARGUMENT;
        if (seed_bytes && (!seeds || !aligned16(seeds))) return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    MixerLayout L;
    mixer_layout(p, n_proj, &L);
    if (p.BH == 0 || p.N == 0) return FLAREPP_OK;  // O is empty
    if (!workspace || ((uintptr_t)workspace % kWsAlign) != 0 || workspace_bytes < L.total)
        return FLAREPP_ERR_WORKSPACE;
    if (overlaps(O, x_bytes, workspace, L.total)) return FLAREPP_ERR_INVALID_ARGUMENT;
    {
        const void* ins[4] = {X, W_in, Wo, seeds};
        const size_t nb[4] = {x_bytes, w_bytes, wo_bytes, seed_bytes};
        if (spans_overlap(ins, nb, 4, workspace, L.total)) return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    if (p.M == 0)  // every decode row has no keys: Y = 0, so O = 0
        return cudaMemsetAsync(O, 0, x_bytes, st) == cudaSuccess ? FLAREPP_OK : FLAREPP_ERR_CUDA;
    char* ws = (char*)workspace;
    int* status = (int*)(ws + p.off_status);
    if (cudaMemsetAsync(status, 0, sizeof(int32_t), st) != cudaSuccess) return FLAREPP_ERR_CUDA;
    auto mark = [&](int i) {
        return !events || cudaEventRecord((cudaEvent_t)events[i], st) == cudaSuccess;
    };
    // the projections go to the workspace, or (training) into `saved` for the backward
    const MixerSaved ms = mixer_saved(p, n_proj);
    void* proj[4];
    for (int i = 0; i < 4; ++i) {
        const int k = i < n_proj ? i : i - 2;
        proj[i] = saved ? saved + ms.off_proj[k] : ws + L.off_proj[k];
    }
    // K, V, K~, V~ = X W_in^T, split into heads (eqs. flarepp_query_synthesis, flarepp_mixer)
    if (!mark(0) ||
        tc_projection(p.B, p.N, p.H, p.D, n_proj, X, W_in, proj, status, st) != cudaSuccess ||
        !mark(1))
        return FLAREPP_ERR_CUDA;
    // the routing chain; the shared variant reads K, V as K~, V~ (App. C.2). A training
    // forward keeps Y and the chain's state in `saved`.
    void* Y = saved ? saved + ms.off_y : ws + L.off_y;
    stt = route_impl(shape, seeds, proj[2], proj[3], proj[0], proj[1], scale, Y, workspace,
                     p.total, stream, nullptr, nullptr, nullptr, 0, false, saved);
    if (stt != FLAREPP_OK) return stt;
    // O = merge(Y) Wo^T
    if (!mark(2) ||
        tc_output_projection(p.B, p.N, p.H, p.D, Y, Wo, O, status, st) != cudaSuccess ||
        !mark(3))
        return FLAREPP_ERR_CUDA;
    return FLAREPP_OK;
}

// Workspace of the mixer's backward: the chain's backward workspace first (its status word at
// offset 0), then dY, the chain's gradients, the transposed weights and the weight
// gradients' float32 partials.
struct MixerBwdLayout {
    size_t off_dy, off_dproj[4], off_wot, off_wint, off_part, total;
};

MixerBwdLayout mixer_bwd_layout(const Plan& p, const BwdPlan& bp, int n_proj) {
    MixerBwdLayout L;
    const size_t tok = (size_t)p.BH * (size_t)p.N * (size_t)p.D * 2;
    const int64_t C = p.H * p.D;
    (void)n_proj;
    size_t off = align_up(bp.total, kWsAlign);
    L.off_dy = off;
    off = align_up(off + tok, kWsAlign);
    for (int i = 0; i < 4; ++i) {
        L.off_dproj[i] = off;
        off = align_up(off + tok, kWsAlign);
    }
    L.off_wot = off;
    off = align_up(off + (size_t)C * (size_t)C * 2, kWsAlign);
    L.off_wint = off;
    off = align_up(off + (size_t)C * 4 * (size_t)C * 2, kWsAlign);
    L.off_part = off;
    const size_t pa = wgrad_plan(p.B, p.N, C, C).part_bytes;
    const size_t pb = wgrad_plan(p.B, p.N, 4 * C, C).part_bytes;
    off = align_up(off + (pa > pb ? pa : pb), kWsAlign);
    L.total = off;
    return L;
}

flarepp_status mixer_bwd_impl(const flarepp_shape* shape, int n_proj, const void* X,
                              const void* W_in, const void* Wo, const void* seeds, float scale,
                              const void* saved, size_t saved_bytes, const void* dO, void* dX,
                              void* dW_in, void* dWo, void* dseeds, void* workspace,
                              size_t workspace_bytes, void* stream) {
    Plan p;
    flarepp_status stt = make_plan(shape, &p);
    if (stt != FLAREPP_OK) return stt;
    if (n_proj != 2 && n_proj != 4) return FLAREPP_ERR_INVALID_ARGUMENT;
    if (p.dtype != FLAREPP_BF16) return FLAREPP_ERR_UNSUPPORTED;
    if (!isfinite(scale)) return FLAREPP_ERR_INVALID_ARGUMENT;
    cudaStream_t st = (cudaStream_t)stream;
    const int64_t C = p.H * p.D;
    const size_t x_bytes = (size_t)p.B * (size_t)p.N * (size_t)C * 2;
    const size_t w_bytes = (size_t)n_proj * (size_t)C * (size_t)C * 2;
    const size_t wo_bytes = (size_t)C * (size_t)C * 2;
    const size_t seed_bytes = (size_t)p.H * (size_t)p.M * (size_t)p.D * 2;
    // every pointer that a non-empty shape needs: present and aligned; outputs disjoint from
    // the inputs
    const void* ins[5] = {X, W_in, Wo, seeds, dO};
    const size_t ib[5] = {x_bytes, w_bytes, wo_bytes, seed_bytes, x_bytes};
    void* outs[4] = {dX, dW_in, dWo, dseeds};
    const size_t ob[4] = {x_bytes, w_bytes, wo_bytes, seed_bytes};
    for (int i = 0; i < 5; ++i)
        if (ib[i] && (!ins[i] || !aligned16(ins[i]))) return FLAREPP_ERR_INVALID_ARGUMENT;
    for (int i = 0; i < 4; ++i) {
        if (ob[i] && (!outs[i] || !aligned16(outs[i]))) return FLAREPP_ERR_INVALID_ARGUMENT;
        if (spans_overlap(ins, ib, 5, outs[i], ob[i])) return FLAREPP_ERR_INVALID_ARGUMENT;
        for (int j = 0; j < i; ++j)
            if (overlaps(outs[i], ob[i], outs[j], ob[j])) return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    const bool work = p.BH && p.N && p.M;
    if (!work) {  // every gradient that exists is zero
        for (int i = 0; i < 4; ++i)
            if (ob[i] && cudaMemsetAsync(outs[i], 0, ob[i], st) != cudaSuccess)
                return FLAREPP_ERR_CUDA;
        return FLAREPP_OK;
    }
    const MixerSaved ms = mixer_saved(p, n_proj);
    if (!saved || !aligned16(saved) || saved_bytes < ms.total) return FLAREPP_ERR_INVALID_ARGUMENT;
    const BwdPlan bp = make_bwd_plan(p);
    const MixerBwdLayout L = mixer_bwd_layout(p, bp, n_proj);
    if (!workspace || ((uintptr_t)workspace % kWsAlign) != 0 || workspace_bytes < L.total)
        return FLAREPP_ERR_WORKSPACE;
    {
        const void* all[9] = {X, W_in, Wo, seeds, dO, saved, dX, dW_in, dWo};
        const size_t nb[9] = {x_bytes, w_bytes, wo_bytes, seed_bytes, x_bytes, ms.total,
                              x_bytes, w_bytes, wo_bytes};
        if (spans_overlap(all, nb, 9, workspace, L.total) ||
            overlaps(dseeds, seed_bytes, workspace, L.total) ||
            overlaps(dseeds, seed_bytes, saved, ms.total))
            return FLAREPP_ERR_INVALID_ARGUMENT;
        for (int i = 0; i < 4; ++i)
            if (overlaps(outs[i], ob[i], saved, ms.total)) return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    char* ws = (char*)workspace;
    int* status = (int*)(ws + bp.off_status);
    const char* sv = (const char*)saved;
    const void* Y = sv + ms.off_y;
    if (cudaMemsetAsync(status, 0, sizeof(int32_t), st) != cudaSuccess) return FLAREPP_ERR_CUDA;
    const void* proj[4];
    for (int i = 0; i < 4; ++i) proj[i] = sv + ms.off_proj[i < n_proj ? i : i - 2];
    void* dY = ws + L.off_dy;
    void* dproj[4];
    for (int i = 0; i < 4; ++i) dproj[i] = ws + L.off_dproj[i];
    void* WoT = ws + L.off_wot;
    void* WinT = ws + L.off_wint;
    float* part = (float*)(ws + L.off_part);
    const int fold = 4 / n_proj;
    cudaError_t e;
    // the weights transposed (W_in repeated for tied projections: K~, V~ use W_K, W_V)
    if ((e = transpose_bf16(Wo, C, C, 1, WoT, st)) != cudaSuccess ||
        (e = transpose_bf16(W_in, n_proj * C, C, fold, WinT, st)) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    // dY = split(dO Wo) (the projections K, V, K~, V~ come from the training forward)
    void* dys[4] = {dY, dY, dY, dY};
    if (tc_projection(p.B, p.N, p.H, p.D, 1, dO, WoT, dys, status, st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    // dWo = dO^T merge(Y)
    WgradSource sdo{0, 1, {dO, dO, dO, dO}};
    WgradSource sy{1, 1, {Y, Y, Y, Y}};
    if (tc_wgrad(p.B, p.N, p.H, p.D, sdo, sy, C, C, C, 1, part, dWo, status, st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    // the chain's backward (App. A.5)
    if (route_bwd(p, bp, seeds, proj[2], proj[3], proj[0], proj[1], scale, Y, dY, sv, dseeds,
                  dproj[2], dproj[3], dproj[0], dproj[1], ws, st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    // dW_in = dP^T X (tied projections fold their two gradients), dX = sum_p dP_p W_p
    WgradSource sdp{1, 4, {dproj[0], dproj[1], dproj[2], dproj[3]}};
    WgradSource sx{0, 1, {X, X, X, X}};
    if (tc_wgrad(p.B, p.N, p.H, p.D, sdp, sx, 4 * C, C, n_proj * C, fold, part, dW_in, status,
                 st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    const void* dps[4] = {dproj[0], dproj[1], dproj[2], dproj[3]};
    if (tc_heads_projection(p.B, p.N, p.H, p.D, 4, dps, WinT, dX, status, st) != cudaSuccess)
        return FLAREPP_ERR_CUDA;
    return FLAREPP_OK;
}

}  // namespace
}  // namespace flarepp

extern "C" {

size_t flarepp_mixer_saved_bytes(const flarepp_shape* shape, int n_proj) {
    flarepp::Plan p;
    if (flarepp::make_plan(shape, &p) != FLAREPP_OK) return 0;
    if ((n_proj != 2 && n_proj != 4) || p.dtype != FLAREPP_BF16) return 0;
    if (p.BH == 0 || p.N == 0 || p.M == 0) return 0;
    return flarepp::mixer_saved(p, n_proj).total;
}

flarepp_status flarepp_mixer_fwd_train(const flarepp_shape* shape, int n_proj, const void* X,
                                       const void* W_in, const void* Wo, const void* seeds,
                                       float scale, void* O, void* saved, size_t saved_bytes,
                                       void* workspace, size_t workspace_bytes, void* stream) {
    flarepp::Plan p;
    const flarepp_status stt = flarepp::make_plan(shape, &p);
    if (stt != FLAREPP_OK) return stt;
    if (p.dtype == FLAREPP_BF16 && p.BH && p.N && p.M) {
        if (n_proj != 2 && n_proj != 4) return FLAREPP_ERR_INVALID_ARGUMENT;
        const size_t need = flarepp::mixer_saved(p, n_proj).total;
        if (!saved || !flarepp::aligned16(saved) || saved_bytes < need)
            return FLAREPP_ERR_INVALID_ARGUMENT;
        if (flarepp::overlaps(saved, need, workspace, workspace_bytes))
            return FLAREPP_ERR_INVALID_ARGUMENT;
    } else {
        saved = nullptr;
    }
    return flarepp::mixer_impl(shape, n_proj, X, W_in, Wo, seeds, scale, O, workspace,
                               workspace_bytes, stream, nullptr, (char*)saved);
}

size_t flarepp_mixer_bwd_workspace_bytes(const flarepp_shape* shape, int n_proj) {
    flarepp::Plan p;
    if (flarepp::make_plan(shape, &p) != FLAREPP_OK) return 0;
    if ((n_proj != 2 && n_proj != 4) || p.dtype != FLAREPP_BF16) return 0;
    if (p.BH == 0 || p.N == 0 || p.M == 0) return 0;
    return flarepp::mixer_bwd_layout(p, flarepp::make_bwd_plan(p), n_proj).total;
}

flarepp_status flarepp_mixer_bwd(const flarepp_shape* shape, int n_proj, const void* X,
                                 const void* W_in, const void* Wo, const void* seeds, float scale,
                                 const void* saved, size_t saved_bytes, const void* dO, void* dX,
                                 void* dW_in, void* dWo, void* dseeds, void* workspace,
                                 size_t workspace_bytes, void* stream) {
    return flarepp::mixer_bwd_impl(shape, n_proj, X, W_in, Wo, seeds, scale, saved, saved_bytes,
                                   dO, dX, dW_in, dWo, dseeds, workspace, workspace_bytes, stream);
}

size_t flarepp_mixer_workspace_bytes(const flarepp_shape* shape, int n_proj) {
    flarepp::Plan p;
    if (flarepp::make_plan(shape, &p) != FLAREPP_OK) return 0;
    if ((n_proj != 2 && n_proj != 4) || p.dtype != FLAREPP_BF16) return 0;
    if (p.BH == 0 || p.N == 0) return 0;
    flarepp::MixerLayout L;
    flarepp::mixer_layout(p, n_proj, &L);
    return L.total;
}

flarepp_status flarepp_mixer_fwd(const flarepp_shape* shape, int n_proj, const void* X,
                                 const void* W_in, const void* Wo, const void* seeds, float scale,
                                 void* O, void* workspace, size_t workspace_bytes, void* stream) {
    return flarepp::mixer_impl(shape, n_proj, X, W_in, Wo, seeds, scale, O, workspace,
                               workspace_bytes, stream);
}

flarepp_status flarepp_mixer_fwd_profiled(const flarepp_shape* shape, int n_proj, const void* X,
                                          const void* W_in, const void* Wo, const void* seeds,
                                          float scale, void* O, void* workspace,
                                          size_t workspace_bytes, void* stream,
                                          void* const* events, int n_events) {
    if (!events || n_events < 4) return FLAREPP_ERR_INVALID_ARGUMENT;
    for (int i = 0; i < 4; ++i)
        if (!events[i]) return FLAREPP_ERR_INVALID_ARGUMENT;
    return flarepp::mixer_impl(shape, n_proj, X, W_in, Wo, seeds, scale, O, workspace,
                               workspace_bytes, stream, events);
}

size_t flarepp_route_saved_bytes(const flarepp_shape* shape) {
    flarepp::Plan p;
    if (flarepp::make_plan(shape, &p) != FLAREPP_OK) return 0;
    if (p.BH == 0 || p.N == 0 || p.M == 0) return 0;
    return flarepp::saved_layout(p).total;
}

flarepp_status flarepp_route_fwd_train(const flarepp_shape* shape, const void* seeds,
                                       const void* Kt, const void* Vt, const void* K,
                                       const void* V, float scale, void* Y, void* saved,
                                       size_t saved_bytes, void* workspace,
                                       size_t workspace_bytes, void* stream) {
    return flarepp::route_fwd_train_impl(shape, seeds, Kt, Vt, K, V, scale, Y, saved,
                                         saved_bytes, workspace, workspace_bytes, stream);
}

size_t flarepp_route_bwd_workspace_bytes(const flarepp_shape* shape) {
    flarepp::Plan p;
    if (flarepp::make_plan(shape, &p) != FLAREPP_OK) return 0;
    return flarepp::make_bwd_plan(p).total;
}

flarepp_status flarepp_route_bwd(const flarepp_shape* shape, const void* seeds, const void* Kt,
                                 const void* Vt, const void* K, const void* V, float scale,
                                 const void* Y, const void* dY, const void* saved,
                                 size_t saved_bytes, void* dseeds, void* dKt, void* dVt,
                                 void* dK, void* dV, void* workspace, size_t workspace_bytes,
                                 void* stream) {
    return flarepp::route_bwd_impl(shape, seeds, Kt, Vt, K, V, scale, Y, dY, saved, saved_bytes,
                                   dseeds, dKt, dVt, dK, dV, workspace, workspace_bytes, stream);
}

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

flarepp_status flarepp_flare_fwd(const flarepp_shape* shape, const void* Q, const void* K,
                                 const void* V, float scale, void* Y, void* workspace,
                                 size_t workspace_bytes, void* stream, float* Z_out) {
    return flarepp::flare_impl(shape, Q, K, V, scale, Y, workspace, workspace_bytes, stream,
                               Z_out);
}

size_t flarepp_route_host_buffer_bytes(const flarepp_shape* shape) {
    flarepp::Plan p;
    if (flarepp::make_plan(shape, &p) != FLAREPP_OK) return 0;
    if (p.BH == 0 || p.N == 0) return 0;
    const flarepp::HostGroups g = flarepp::host_groups(p);
    flarepp::HostLayout L;
    if (!flarepp::host_layout(shape, p, g, &L)) return 0;
    return L.total;
}

flarepp_status flarepp_flare_fwd_host(const flarepp_shape* shape, const void* Q, const void* K,
                                      const void* V, float scale, void* Y, void* device_buffer,
                                      size_t device_buffer_bytes, void* stream) {
    return flarepp::route_host_impl(shape, Q, K, V, K, V, scale, Y, device_buffer,
                                    device_buffer_bytes, stream, true);
}

flarepp_status flarepp_route_fwd_host(const flarepp_shape* shape, const void* seeds,
                                      const void* Kt, const void* Vt, const void* K,
                                      const void* V, float scale, void* Y, void* device_buffer,
                                      size_t device_buffer_bytes, void* stream) {
    return flarepp::route_host_impl(shape, seeds, Kt, Vt, K, V, scale, Y, device_buffer,
                                    device_buffer_bytes, stream);
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

void flarepp_test_wait_fault(int kernel, int64_t ring_item, uint64_t wait_ns) {
    flarepp::set_tc_test_fault(kernel, ring_item, wait_ns);
}

}  // extern "C"
