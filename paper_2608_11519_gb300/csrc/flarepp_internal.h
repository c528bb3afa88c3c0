// Internal declarations shared by the libflarepp translation units (not installed).
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "flarepp.h"

namespace flarepp {

constexpr int kNumSMs = 152;  // GB300: two dies of 76 SMs
constexpr size_t kWsAlign = 256;  // alignment of every workspace sub-buffer

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
inline int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Which kernels a shape runs on.
enum Path : int {
    kPathSimt = 0,  // CUDA-core kernels: the float32 dtype path
    kPathTc = 1,    // tcgen05 / TMEM / TMA kernels: the bf16 dtype path
};

// Everything a launch needs, derived from the shape alone.
struct Plan {
    int64_t B, H, N, M, D, BH;
    int dtype;
    int path;
    // split-N encode: tokens [c * chunk_len, min(N, (c + 1) * chunk_len)) form chunk c
    int64_t chunk_len, nchunk;
    int64_t m_tile, n_mtiles;  // CUDA-core encode: routes per CTA and route tiles per head
    int64_t n_groups;          // tensor-core encode: route groups per head
    int64_t tc_group;          // tensor-core encode: routes per group (4 or 2 tiles of 128)
    int64_t sub_per_chunk;     // partial slots per chunk (1 CUDA-core, 4 tensor-core)
    // workspace layout (byte offsets from the workspace base, each 256-byte aligned)
    size_t off_status;                    // int32 device status word (FLAREPP_OK or _TIMEOUT)
    size_t off_overflow;                  // int32 x 3: the tensor-core kernels' overflow words
    size_t off_pmax, off_psum, off_pacc;  // partials [BH][nchunk*sub][M] f32 x2, (...)[D] f32
    size_t off_q32, off_z32;              // Q, Z float32 [BH][M][D]
    size_t off_qop, off_zop;              // bf16 MMA operand copies of Q, Z [BH][M][D]
    size_t off_qlo;                       // bf16 lo part of Q's operand, Q - qop [BH][M][D]
    size_t off_seedneg;                   // bf16 -seeds [H][M][D] (used when scale < 0)
    size_t total;
};

// Launch `kernel` on `st` with programmatic stream serialization: its blocks may start while
// the kernel before it on the stream finishes, and wait for it at their pdl_wait (the kernels
// of the chain call it before touching memory that the previous kernel writes or reads).
template <typename... Params, typename... Args>
cudaError_t launch_pdl(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Raise the dynamic shared-memory limit of kernel `func` to `bytes` on the current device,
// once per (kernel, device): the attribute is per device, so a process that launches on
// several GPUs sets it on each (flarepp_api.cu).
cudaError_t ensure_smem_limit(const void* func, int bytes);

// Fill `p` for `s` (plan.cu); returns FLAREPP_OK or the validation error for the shape itself.
flarepp_status make_plan(const flarepp_shape* s, Plan* p);

// The state a training forward keeps for the backward (App. A.5), in a caller buffer:
// float32 Q and Z [BH][M][D] and the log-normalisers of the three calls in base 2,
// L = log2 sum_j 2^(scale * log2(e) <a, b_j>): L1, L2 [BH][M] and L3 [BH][N].
struct SavedLayout {
    size_t off_q, off_z, off_l1, off_l2, off_l3, total;
};
SavedLayout saved_layout(const Plan& p);

// The backward's plan: the split-N route passes (chunks of tokens) and its workspace. On
// the CUDA-core path a route pass gives one thread per route (m_tile routes per CTA); on
// the tensor-core path a work unit is a group of up to 512 routes and a chunk of tokens,
// and chunk_len is a multiple of 192 tokens (whole items of every size: 32, 48, 64).
struct BwdPlan {
    int path;                   // kPathSimt or kPathTc
    int64_t m_tile, n_mtiles;   // CUDA-core route passes: routes per CTA, route tiles per head
    int64_t chunk_len, nchunk;  // tokens per chunk and chunks per head
    size_t off_status;          // int32 device status word
    size_t off_pa, off_pb;      // per-chunk partial sums [BH][nchunk][M][D] f32
    size_t off_dz, off_dq;      // dZ, dQ [BH][M][D] f32
    size_t off_d1, off_d2;      // c = <dO, O> of calls 1 and 2 [BH][M] f32
    size_t off_d3;              // c of call 3 [BH][N] f32 (+ 256 bytes of slack)
    size_t off_qb, off_zb;      // tensor-core path: bf16 MMA operands Q, Z [BH][M][D]
    size_t off_dzb, off_dqb;    // ... and dZ, dQ
    size_t off_qlo;             // ... and Q's lo part, Q - bf16(Q) (D <= 32)
    size_t off_w;               // ... and the merged T23 pass's w dZ [BH][M][D] bf16
    size_t off_rb, off_flags;   // its shift R [BH] f32 and fallback flags [BH] int32
    size_t off_rpart;           // range partials [BH][kRangeParts + 2] f32
    size_t total;
};
constexpr int kRangeParts = 128;  // token slices of the merged pass's range reduction
BwdPlan make_bwd_plan(const Plan& p);

// ---- CUDA-core kernels (simt_kernels.cuh, instantiated in simt_f32.cu), float32 inputs
// Encode one call over all chunks: call 1 takes the seeds ([H][M][D]), call 2 takes Q32
// from the workspace. Writes the chunk partials.
cudaError_t simt_encode_f32(const Plan& p, int call, const void* k, const void* v,
                            const void* seeds, float scale, char* ws, cudaStream_t st);
// Decode (call 3) on CUDA cores: Y = SDPA(K, Q32, Z32); also the base-2 log-normaliser of
// each token's row into `lse` [BH][N] when it is not null.
cudaError_t simt_decode_f32(const Plan& p, const void* K, float scale, void* Y, char* ws,
                            cudaStream_t st, float* lse = nullptr);

// ---- backward (bwd.cu): the passes of App. A.5. f32 inputs run on CUDA cores, bf16 inputs
// on the tensor-core passes of tc_bwd.cu. `saved` is the training forward's state, `ws`
// the backward workspace; outputs in the input dtype.
cudaError_t route_bwd(const Plan& p, const BwdPlan& bp, const void* seeds, const void* Kt,
                      const void* Vt, const void* K, const void* V, float scale, const void* Y,
                      const void* dY, const char* saved, void* dseeds, void* dKt, void* dVt,
                      void* dK, void* dV, char* ws, cudaStream_t st);

// ---- split-N combine (combine.cu)
// Stable log-sum-exp merge of the chunk partials into Q32 (call 1) or Z32 (call 2), plus
// the bf16 MMA operand copy when the tensor-core path consumes it (negated when
// `negate`, which together with negated seeds turns a negative scale into |scale|).
// The base-2 log-normaliser of each merged row goes to `lse` [BH][M] when it is not null.
// With `lo` (call 1, tensor-core path) the merge also writes bf16(Q' - bf16(Q')), Q' the
// possibly negated Q, to the workspace's lo operand.
cudaError_t combine(const Plan& p, int call, char* ws, bool negate, cudaStream_t st,
                    float* lse = nullptr, bool lo = false);
// dst = -src elementwise (bf16; exact)
cudaError_t negate_bf16(const void* src, void* dst, int64_t n, cudaStream_t st);

// ---- tensor-core backward passes (tc_bwd.cu), bf16 inputs
// Operands of one pass: its A tiles and item tiles (bf16 [z][rows][D]; an unused third
// entry may repeat a used one), the row and column statistics, and its outputs (partial
// sums of the route-row passes, bf16 gradients of the token-row passes).
struct TcBwdOperands {
    const void* a[3];
    const void* i[3];
    const float* Lrow;
    const float* crow;
    const float* Lcol;
    const float* ccol;
    float* pa;
    float* pb;
    void* out0;
    void* out1;
    const float* Rb = nullptr;  // T23C: the shift R of each (b, h)
    const int* flags = nullptr;  // when set, only the (b, h) with flags[bh] == want run
    int want = 0;
    // Q's bf16 lo operand (Q - bf16(Q)) for the hi/lo score products of R3, R2, T23 and T23C
    // at D <= 32, or null (plain bf16 Q)
    const void* lo = nullptr;
};
// pass: 0 = R3, 1 = R2, 2 = R1 (route rows), 3 = T23, 4 = T1 (token rows), 5 = T23C (T23
// with its two dP products merged; D = 16 and 32)
cudaError_t tc_bwd_pass(const Plan& p, const BwdPlan& bp, int pass, const TcBwdOperands& o,
                        float scale, int* status, cudaStream_t st);

// ---- the mixer's pointwise projections (tc_gemm.cu), bf16
// X [B][N][C] times W_in [P*C][C] (out x in) into the P tensors outs[p] [B][H][N][D]
// (C = H * D; P = 4: K, V, K~, V~; P = 2: K, V).
cudaError_t tc_projection(int64_t B, int64_t N, int64_t H, int64_t D, int P, const void* X,
                          const void* W_in, void* const* outs, int* status, cudaStream_t st);
// merge(Y) times Wo [C][C] (out x in) into O [B][N][C], Y read head by head [B][H][N][D].
cudaError_t tc_output_projection(int64_t B, int64_t N, int64_t H, int64_t D, const void* Y,
                                 const void* Wo, void* O, int* status, cudaStream_t st);
// n_a head-layout tensors As[p] [B][H][N][D] side by side (channel p*C + h*D + d) times
// W [C][n_a * C] (out x in) into O [B][N][C].
cudaError_t tc_heads_projection(int64_t B, int64_t N, int64_t H, int64_t D, int n_a,
                                const void* const* As, const void* W, void* O, int* status,
                                cudaStream_t st);

// ---- the mixer's weight gradients (tc_wgrad.cu), bf16
// A channel source: `heads` = 1 for n tensors [B][H][N][D] side by side (channel p*C + h*D + d),
// 0 for one matrix [B][N][C].
struct WgradSource {
    int heads;
    int n;
    const void* t[4];
};
struct WgradPlan {
    int NT;
    int64_t row_tiles, col_tiles, chunk_len, chunks_per_b, n_chunks;
    size_t part_bytes;  // float32 partials [n_chunks][R][Cc]
};
WgradPlan wgrad_plan(int64_t B, int64_t N, int64_t R, int64_t Cc);
// dW [R_out][Cc] (bf16) = sum over tokens of A(t, r) B(t, c) for r < R, c < Cc, the rows
// r + k * R_out (k < fold) added into row r; `part` holds the plan's partials.
cudaError_t tc_wgrad(int64_t B, int64_t N, int64_t H, int64_t D, const WgradSource& a,
                     const WgradSource& b, int64_t R, int64_t Cc, int64_t R_out, int fold,
                     float* part, void* dW, int* status, cudaStream_t st);
// dst [Cc][rep * R] = the transpose of src [R][Cc] repeated rep times along its columns
cudaError_t transpose_bf16(const void* src, int64_t R, int64_t Cc, int rep, void* dst,
                           cudaStream_t st);
// dst += src, elementwise over n bf16 values (float32 sum, rounded once)
cudaError_t add_bf16(void* dst, const void* src, int64_t n, cudaStream_t st);

// ---- tensor-core kernels (tc_kernels.cu), bf16 inputs
// Encode call 1 (A = seeds) or call 2 (A = Q operand) into the chunk partials. With `lo`
// (call 2, D <= 32) the scores take Q as its hi and lo bf16 operands.
cudaError_t tc_encode(const Plan& p, int call, const void* k, const void* v, const void* seeds,
                      float scale, char* ws, cudaStream_t st, bool lo = false);
// Test hook of the bounded waits: until reset (kernel = 0), the launches of one tensor-core
// chain kernel (1, 2: the encode of call 1 or 2; 3: the decode) wait at most wait_ns at each
// barrier, and CTA 0's producer never loads ring item `ring_item` (so that a wait runs out).
void set_tc_test_fault(int kernel, int64_t ring_item, uint64_t wait_ns);
// The wait bound and withheld ring item of a launch of tensor-core kernel `kernel` (1, 2:
// encode; 3: decode; 4 + p: backward pass p): the hook's setting for that kernel, else 2 s and
// none.
void test_fault_for(int kernel, uint64_t* wait_ns, int64_t* ring_item);
// Rows per tensor-core work unit (route group of the encode, token group of the decode).
int64_t tc_group_rows(int64_t D);
int64_t tc_encode_item_rows(int64_t D);  // tokens per item of the tensor-core encode
// Decode call 3: Y = SDPA(K, Q, Z) from the Q and Z operand copies; also each token's
// base-2 log-normaliser into `lse` [BH][N] when it is not null. With `lo` (D <= 32) the
// scores take Q as its hi and lo bf16 operands.
cudaError_t tc_decode(const Plan& p, const void* K, float scale, void* Y, char* ws,
                      cudaStream_t st, float* lse = nullptr, bool lo = false);

}  // namespace flarepp
