/*
 * libflarepp -- the FLARE++ routing chain on one GB300 (sm_103a).
 *
 * For every batch element b and head h the library computes three scaled-dot-product
 * attention calls (FLARE++ paper, Sec. 3.2, eqs. flarepp_dynamic_query and flarepp_mixer;
 * SDPA as in Sec. 2, eq. sdpa_definition):
 *
 *   call 1  Q = SDPA(seeds_h, Kt, Vt)   softmax over the N tokens   -> Q [M, D]
 *   call 2  Z = SDPA(Q, K, V)           softmax over the N tokens   -> Z [M, D]
 *   call 3  Y = SDPA(K, Q, Z)           softmax over the M routes   -> Y [N, D]
 *
 * with SDPA(A, B, C) = softmax(scale * A B^T) C. Calls 1 and 2 run as a split-N encode
 * (each CTA reduces a chunk of tokens to online-softmax partials) followed by the stable
 * log-sum-exp merge of App. A.3, the single-GPU form of the token-sharded encoder of
 * Sec. 3.3 / eq. distributed_flare_encoder. Call 3 runs as an N-tiled decode.
 *
 * Conventions shared by every entry point
 *   - Layout: dense row-major, D innermost. seeds [H, M, D]; Kt, Vt, K, V, Y [B, H, N, D].
 *     Inputs and Y share one element type, chosen by flarepp_shape.dtype.
 *   - Pointers: device pointers (or managed memory), each 16-byte aligned. The caller owns
 *     every buffer; the library keeps no pointer after a call returns and allocates no
 *     device memory. Y must not overlap any input or the workspace, nor the workspace an
 *     input (FLAREPP_ERR_INVALID_ARGUMENT).
 *   - Stream: all work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and the call returns without synchronising. The workspace must stay untouched
 *     until that work has finished.
 *   - Errors: arguments are checked before anything is launched; on a non-OK status nothing
 *     has been enqueued, except FLAREPP_ERR_CUDA, which reports a failed launch. No C++
 *     exception crosses this interface and nothing is printed.
 *   - Supported: D in {16, 32, 64}; 0 <= M <= 2048; B, H, N >= 0; finite scale.
 *     N = 0 or B*H = 0 is a no-op. M = 0 writes Y = 0: every decode row then has no keys,
 *     and an attention row with no keys outputs 0 (App. A.3).
 *   - Threads: entry points may be called from several host threads at once (on distinct
 *     workspaces and outputs).
 */
#ifndef FLAREPP_H
#define FLAREPP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define FLAREPP_API __attribute__((visibility("default")))
#else
#define FLAREPP_API
#endif

typedef enum {
    FLAREPP_F32 = 0,  /* inputs and Y are float32; the path computes in float32 */
    FLAREPP_BF16 = 1  /* inputs and Y are bfloat16; tensor-core products, float32 accumulate */
} flarepp_dtype;

typedef enum {
    FLAREPP_OK = 0,
    FLAREPP_ERR_INVALID_ARGUMENT = 1, /* null/misaligned pointer, negative size, NaN/inf scale,
                                         overlapping buffers, bad dtype */
    FLAREPP_ERR_UNSUPPORTED = 2,      /* a valid shape outside the supported set (D, M limits) */
    FLAREPP_ERR_WORKSPACE = 3,        /* workspace missing, misaligned or too small */
    FLAREPP_ERR_CUDA = 4,             /* a CUDA call or kernel launch failed */
    FLAREPP_ERR_TIMEOUT = 5           /* reserved: a bounded device wait gave up */
} flarepp_status;

typedef struct {
    int64_t B; /* batch elements */
    int64_t H; /* heads */
    int64_t N; /* tokens */
    int64_t M; /* routes (latent slots) */
    int64_t D; /* head width */
    int32_t dtype; /* flarepp_dtype */
} flarepp_shape;

/*
 * Bytes of device workspace that flarepp_route_fwd needs for `shape` (a function of the
 * shape alone). Returns 0 when the shape is invalid or needs none. The workspace holds the
 * split-N partials (running max, sum and weighted value sum per chunk and route) and the
 * routing queries Q and latents Z of calls 1 and 2.
 */
FLAREPP_API size_t flarepp_route_workspace_bytes(const flarepp_shape* shape);

/*
 * The routing chain (Sec. 3.2, eqs. flarepp_dynamic_query and flarepp_mixer).
 *   seeds      [H, M, D]     learned route seeds, shared by all b (App. A.1)
 *   Kt, Vt     [B, H, N, D]  keys and values of the query-synthesis call
 *   K, V       [B, H, N, D]  keys and values of the gather/scatter pair
 *   scale      softmax temperature of all three calls; 1/sqrt(D) in the paper
 *   Y          [B, H, N, D]  output, written in full
 *   workspace  >= flarepp_route_workspace_bytes(shape) bytes, 256-byte aligned
 *   stream     cudaStream_t to enqueue on
 */
FLAREPP_API flarepp_status flarepp_route_fwd(const flarepp_shape* shape, const void* seeds, const void* Kt,
                                 const void* Vt, const void* K, const void* V, float scale,
                                 void* Y, void* workspace, size_t workspace_bytes, void* stream);

/*
 * flarepp_route_fwd that also copies the intermediates out, so each call of the chain can be
 * checked on its own: Q_out and Z_out are float32 [B, H, M, D] device buffers (each may be
 * NULL). Same rules and errors as flarepp_route_fwd.
 */
FLAREPP_API flarepp_status flarepp_route_fwd_debug(const flarepp_shape* shape, const void* seeds,
                                       const void* Kt, const void* Vt, const void* K,
                                       const void* V, float scale, void* Y, void* workspace,
                                       size_t workspace_bytes, void* stream, float* Q_out,
                                       float* Z_out);

/*
 * flarepp_route_fwd that also records six caller-created CUDA events (cudaEvent_t) on
 * `stream` around its stages, so a caller can time each kernel of the chain on the stream
 * it runs on: events[0] before the call-1 encode, [1] after it, [2] after the call-1
 * combine, [3] after the call-2 encode, [4] after the call-2 combine, [5] after the
 * call-3 decode. n_events must be >= 6 and no event may be NULL (else
 * FLAREPP_ERR_INVALID_ARGUMENT). On degenerate shapes (N, M or B*H zero) no event is
 * recorded. Otherwise identical to flarepp_route_fwd.
 */
FLAREPP_API flarepp_status flarepp_route_fwd_profiled(const flarepp_shape* shape,
                                                      const void* seeds, const void* Kt,
                                                      const void* Vt, const void* K,
                                                      const void* V, float scale, void* Y,
                                                      void* workspace, size_t workspace_bytes,
                                                      void* stream, void* const* events,
                                                      int n_events);

/*
 * FLARE, the fixed-query form of the routing (Sec. 3, eq. prelim_flare_sdpa): per (b, h),
 *   Z = SDPA(Q_h, K, V)   (softmax over the N tokens, one row per route)
 *   Y = SDPA(K, Q_h, Z)   (softmax over the M routes, one row per token)
 * with learned queries Q_h shared by the batch: the routing chain without its first call.
 *   shape: as for flarepp_route_fwd (M routes per head); workspace: at least
 *     flarepp_route_workspace_bytes(shape) bytes, 256-byte aligned.
 *   Q: [H, M, D] in the input dtype. K, V, Y: [B, H, N, D]. Same alignment, aliasing and
 *     scale rules as flarepp_route_fwd (Y must not overlap K, V, Q or the workspace).
 *   Z_out: NULL, or float32 [B, H, M, D] device memory that receives Z.
 * Errors and the device status word: as flarepp_route_fwd.
 */
FLAREPP_API flarepp_status flarepp_flare_fwd(const flarepp_shape* shape, const void* Q,
                                             const void* K, const void* V, float scale, void* Y,
                                             void* workspace, size_t workspace_bytes,
                                             void* stream, float* Z_out);

/*
 * Bytes of device memory that flarepp_route_fwd_host needs for `shape` (its workspace plus
 * device copies of the inputs and of Y), or 0 for an invalid shape or an empty Y.
 */
FLAREPP_API size_t flarepp_route_host_buffer_bytes(const flarepp_shape* shape);

/*
 * The routing chain of flarepp_route_fwd (Sec. 3.2, eqs. flarepp_dynamic_query and
 * flarepp_mixer) on HOST buffers: copies the inputs to the device, runs the chain and copies
 * Y back, with the copies overlapped with the computation. The (b, h) slices of the chain are
 * independent, so the heads are processed in up to eight groups: while the chain of one group
 * runs on `stream`, the next group's inputs are copied in on a second stream and the previous
 * group's Y is copied out on a third.
 *   seeds, Kt, Vt, K, V, Y: host pointers, same layouts and dtypes as flarepp_route_fwd. The
 *     copies overlap the kernels only when the host memory is page-locked (pinned). Passing
 *     Kt == K and Vt == V (the shared-projection variant, App. cost_model) copies them once.
 *   device_buffer: caller-owned device memory of at least flarepp_route_host_buffer_bytes
 *     bytes, 256-byte aligned (else FLAREPP_ERR_WORKSPACE). It starts with the workspace, so
 *     flarepp_route_device_status(shape, device_buffer, ...) reports a timeout in any group.
 *   Streams: the second and third streams and the events that order them are created by the
 *     call and released at its end; CUDA frees them once their work has finished.
 *   Asynchronous: everything is ordered after the work already on `stream`, and later work
 *     on `stream` is ordered after the last copy into Y. The host buffers must stay valid
 *     (and Y unread) until then.
 *   Errors: as flarepp_route_fwd, plus FLAREPP_ERR_CUDA if a stream or event cannot be
 *     created. An empty Y (N or B*H zero) returns FLAREPP_OK without any work.
 */
FLAREPP_API flarepp_status flarepp_route_fwd_host(const flarepp_shape* shape, const void* seeds,
                                                  const void* Kt, const void* Vt, const void* K,
                                                  const void* V, float scale, void* Y,
                                                  void* device_buffer,
                                                  size_t device_buffer_bytes, void* stream);

/*
 * flarepp_flare_fwd (FLARE with the learned queries Q [H, M, D]) on HOST buffers Q, K, V, Y,
 * with the same head groups and overlapped copies as flarepp_route_fwd_host (K and V are
 * copied once). device_buffer: at least flarepp_route_host_buffer_bytes(shape) bytes,
 * 256-byte aligned. Asynchronous and errors as flarepp_route_fwd_host.
 */
FLAREPP_API flarepp_status flarepp_flare_fwd_host(const flarepp_shape* shape, const void* Q,
                                                  const void* K, const void* V, float scale,
                                                  void* Y, void* device_buffer,
                                                  size_t device_buffer_bytes, void* stream);

/*
 * flarepp_route_fwd without a caller-provided workspace. The paper has no counterpart: this
 * entry point exists for callers that cannot allocate device memory when they call the
 * chain. Examples are a plugin whose host application owns all device memory, and a
 * latency-critical loop where cudaMalloc or cudaFree would synchronise the device.
 * Inputs and Y are the caller's, exactly as in flarepp_route_fwd.
 *   - Scratch: a fixed 64 MiB device array inside the library, held by every GPU that
 *     loads it until the process exits. A shape whose flarepp_route_workspace_bytes
 *     exceeds 64 MiB returns FLAREPP_ERR_WORKSPACE and enqueues nothing.
 *   - No allocation: no cudaMalloc, cudaFree or other allocating call is made.
 *   - First call per device: it looks up the array's device address (cudaGetSymbolAddress
 *     with that device current) and caches it. Make that first call before any stream
 *     capture.
 *   - Device: the call uses the array of the current device, so `stream` must belong to the
 *     current device; a stream of another device returns FLAREPP_ERR_INVALID_ARGUMENT.
 *   - Sharing: every call on a device shares the one array, and the array keeps the last
 *     call's contents. Each call clears the status word and writes all the scratch it
 *     reads. Calls whose work overlaps on the GPU (other streams, other host threads) race
 *     on the array and corrupt each other's results. Serialise them.
 *   - The device status word of these calls lives in the array, so
 *     flarepp_route_device_status, which reads a caller's workspace, cannot report it.
 */
FLAREPP_API flarepp_status flarepp_route_fwd_noalloc(const flarepp_shape* shape,
                                                     const void* seeds, const void* Kt,
                                                     const void* Vt, const void* K,
                                                     const void* V, float scale, void* Y,
                                                     void* stream);

/*
 * The FLARE++ token-mixing layer (Fig. 1; eqs. flarepp_query_synthesis, flarepp_mixer): the
 * pointwise projections K, V, K~, V~ = X W_in^T (split into H heads of width D, C = H * D),
 * the routing chain, and O = merge(Y) Wo^T, where merge places the heads side by side.
 *   shape: B, H, N (tokens), M (routes), D and dtype; bf16 only (FLAREPP_ERR_UNSUPPORTED for
 *     float32).
 *   n_proj: 4 (K, V, K~, V~) or 2 (K, V; the shared-projection variant of App. C.2, which
 *     uses K, V as K~, V~).
 *   X: [B, N, C]; W_in: [n_proj * C, C], out x in (row block 0 is W_K, then W_V, W_K~, W_V~);
 *     Wo: [C, C], out x in; seeds: [H, M, D]; O: [B, N, C]. Device pointers, 16-byte
 *     aligned; neither O nor the workspace may overlap an input, nor O the workspace. No
 *     biases.
 *   workspace: flarepp_mixer_workspace_bytes(shape, n_proj) bytes, 256-byte aligned; it holds
 *     the chain's workspace (its status word at offset 0, read by
 *     flarepp_route_device_status), the projections and Y.
 * Degenerate shapes: N or B*H zero leave O (empty) alone; M = 0 writes O = 0.
 * Errors: FLAREPP_ERR_INVALID_ARGUMENT, FLAREPP_ERR_UNSUPPORTED, FLAREPP_ERR_WORKSPACE,
 * FLAREPP_ERR_CUDA, as for flarepp_route_fwd. Enqueued on `stream`.
 */
FLAREPP_API size_t flarepp_mixer_workspace_bytes(const flarepp_shape* shape, int n_proj);
FLAREPP_API flarepp_status flarepp_mixer_fwd(const flarepp_shape* shape, int n_proj,
                                             const void* X, const void* W_in, const void* Wo,
                                             const void* seeds, float scale, void* O,
                                             void* workspace, size_t workspace_bytes,
                                             void* stream);

/*
 * flarepp_mixer_fwd that also records four caller-created CUDA events (cudaEvent_t) on
 * `stream`: events[0] before the input projection, [1] after it, [2] after the routing chain,
 * [3] after the output projection. n_events must be >= 4 and no event may be NULL (else
 * FLAREPP_ERR_INVALID_ARGUMENT); on degenerate shapes no event is recorded.
 */
FLAREPP_API flarepp_status flarepp_mixer_fwd_profiled(const flarepp_shape* shape, int n_proj,
                                                      const void* X, const void* W_in,
                                                      const void* Wo, const void* seeds,
                                                      float scale, void* O, void* workspace,
                                                      size_t workspace_bytes, void* stream,
                                                      void* const* events, int n_events);

/*
 * Training the mixer layer. flarepp_mixer_fwd_train is flarepp_mixer_fwd that also fills
 * `saved` (flarepp_mixer_saved_bytes(shape, n_proj) bytes of device memory, 16-byte aligned,
 * disjoint from the workspace; layout private) with the chain's saved state, Y and the
 * n_proj projections (which the forward writes there instead of into its workspace).
 * flarepp_mixer_bwd then computes, for the output gradient dO [B, N, C]:
 *   dX [B, N, C], dW_in [n_proj * C, C], dWo [C, C] (both out x in, like the weights) and
 *   dseeds [H, M, D],
 * all bf16, written (not accumulated): dO through the output projection (dWo = dO^T merge(Y),
 * dY = split(dO Wo)), the chain's backward (App. A.5), then the projections' backward
 * (dW_in = dP^T X, dX = dP W_in, the gradients of tied projections added for n_proj = 2).
 * The projections are read from `saved`. workspace: flarepp_mixer_bwd_workspace_bytes(shape,
 * n_proj) bytes, 256-byte aligned (its first 4 bytes are the device status word). Outputs
 * must be 16-byte aligned and disjoint from each other, from the inputs and from `saved`;
 * the workspace must be disjoint from all of them. Degenerate
 * shapes (N, M or B*H zero) write zeros to every non-empty gradient. Errors as for
 * flarepp_mixer_fwd.
 */
FLAREPP_API size_t flarepp_mixer_saved_bytes(const flarepp_shape* shape, int n_proj);
FLAREPP_API flarepp_status flarepp_mixer_fwd_train(const flarepp_shape* shape, int n_proj,
                                                   const void* X, const void* W_in,
                                                   const void* Wo, const void* seeds,
                                                   float scale, void* O, void* saved,
                                                   size_t saved_bytes, void* workspace,
                                                   size_t workspace_bytes, void* stream);
FLAREPP_API size_t flarepp_mixer_bwd_workspace_bytes(const flarepp_shape* shape, int n_proj);
FLAREPP_API flarepp_status flarepp_mixer_bwd(const flarepp_shape* shape, int n_proj,
                                             const void* X, const void* W_in, const void* Wo,
                                             const void* seeds, float scale, const void* saved,
                                             size_t saved_bytes, const void* dO, void* dX,
                                             void* dW_in, void* dWo, void* dseeds,
                                             void* workspace, size_t workspace_bytes,
                                             void* stream);

/*
 * Bytes of the state a training forward keeps for the backward (App. A.5): float32 Q and Z
 * [B, H, M, D] and the base-2 log-normalisers of the three calls,
 * L = log2 sum_j 2^(scale * log2(e) <a, b_j>), for calls 1 and 2 [B, H, M] and call 3
 * [B, H, N]. 0 for an invalid or unsupported shape and for N, M or B*H zero.
 */
FLAREPP_API size_t flarepp_route_saved_bytes(const flarepp_shape* shape);

/*
 * flarepp_route_fwd that also fills `saved` (device memory, 16-byte aligned, at least
 * flarepp_route_saved_bytes(shape) bytes, disjoint from the inputs, Y and the workspace;
 * FLAREPP_ERR_INVALID_ARGUMENT otherwise) with the state flarepp_route_bwd reads. The
 * layout of `saved` is private to the library; the caller only keeps it until the backward.
 * On degenerate shapes `saved` is not touched and may be NULL.
 */
FLAREPP_API flarepp_status flarepp_route_fwd_train(const flarepp_shape* shape,
                                                   const void* seeds, const void* Kt,
                                                   const void* Vt, const void* K, const void* V,
                                                   float scale, void* Y, void* saved,
                                                   size_t saved_bytes, void* workspace,
                                                   size_t workspace_bytes, void* stream);

/* Workspace bytes flarepp_route_bwd needs for `shape` (0: none needed or shape invalid). */
FLAREPP_API size_t flarepp_route_bwd_workspace_bytes(const flarepp_shape* shape);

/*
 * Backward of the routing chain (App. A.5): for the output gradient dY, the gradients of
 * the seeds and of Kt, Vt, K, V. Each SDPA is differentiated from its saved output and
 * log-normaliser (P = exp(S - L), c = <dO, O>, dV = P^T dO, dS = P o (dO V^T - c),
 * dK = s dS^T Q, dQ = s dS K); the decoder's gradient of Q is added to the encoder's before
 * call 1's backward, and the seeds' gradient is summed over the batch.
 *   seeds, Kt, Vt, K, V, scale: the forward's inputs (device pointers, as flarepp_route_fwd).
 *   Y: the forward's output [B, H, N, D]; dY: its gradient [B, H, N, D]; both input dtype.
 *   saved: what flarepp_route_fwd_train wrote for these inputs (saved_bytes as there).
 *   dseeds [H, M, D], dKt, dVt, dK, dV [B, H, N, D]: outputs in the input dtype, written
 *     (not accumulated), 16-byte aligned, disjoint from each other and from every input.
 *   workspace: device memory, 256-byte aligned, flarepp_route_bwd_workspace_bytes(shape)
 *     bytes, disjoint from every input, `saved` and the outputs; its first 4 bytes are the
 *     device status word (flarepp_route_device_status).
 * Degenerate shapes (N, M or B*H zero) write zeros to every non-empty output. Errors:
 * FLAREPP_ERR_INVALID_ARGUMENT (a missing, misaligned or overlapping pointer, too small a
 * saved buffer, non-finite scale), FLAREPP_ERR_UNSUPPORTED (as flarepp_route_fwd),
 * FLAREPP_ERR_WORKSPACE, FLAREPP_ERR_CUDA. Enqueued on `stream`; no host synchronisation.
 */
FLAREPP_API flarepp_status flarepp_route_bwd(const flarepp_shape* shape, const void* seeds,
                                             const void* Kt, const void* Vt, const void* K,
                                             const void* V, float scale, const void* Y,
                                             const void* dY, const void* saved,
                                             size_t saved_bytes, void* dseeds, void* dKt,
                                             void* dVt, void* dK, void* dV, void* workspace,
                                             size_t workspace_bytes, void* stream);

/*
 * The device status word that the last flarepp_route_fwd* call on `workspace` (for the same
 * shape) left behind: FLAREPP_OK, or FLAREPP_ERR_TIMEOUT when a bounded wait inside a
 * tensor-core kernel gave up (the kernel then stops early and its outputs are invalid).
 * Copies 4 bytes to *status_out (host memory) on `stream` and synchronises that stream.
 */
FLAREPP_API flarepp_status flarepp_route_device_status(const flarepp_shape* shape,
                                                       const void* workspace, void* stream,
                                                       int32_t* status_out);

/*
 * Test hook of the bounded waits; the paper has no counterpart. It lets a test make a wait
 * inside a tensor-core kernel run out without faulting or hanging the GPU.
 *   kernel: which launch of later calls it applies to: 1 or 2, the encode of call 1 or 2;
 *     3, the decode; 4 + p, pass p of flarepp_route_bwd's tensor-core passes (0: the route
 *     pass of call 3, 1: of call 2, 2: of call 1, 3: the token pass of calls 2 and 3, 4: of
 *     call 1, 5: the merged token pass of calls 2 and 3); 0 turns the hook off (the
 *     default).
 *   ring_item: the index, in the order it is loaded, of an item of CTA 0's ring of K/V (or
 *     Q/Z) tiles that the kernel's load warp then never loads, so that the waits for it run
 *     out (-1: none).
 *   wait_ns: the bound of every wait of that launch (0: the default of 2 s).
 * Process-wide state, for tests only: it applies to every later call from any thread until it
 * is turned off. A launch whose wait ran out stops early and records FLAREPP_ERR_TIMEOUT in
 * the device status word (flarepp_route_device_status); its outputs are invalid.
 */
FLAREPP_API void flarepp_test_wait_fault(int kernel, int64_t ring_item, uint64_t wait_ns);

/* Static description of a status code (never NULL). */
FLAREPP_API const char* flarepp_status_string(flarepp_status status);

/* Library version string, e.g. "0.1.0". */
FLAREPP_API const char* flarepp_version(void);

#ifdef __cplusplus
}
#endif
#endif /* FLAREPP_H */
