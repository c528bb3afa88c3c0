// Internal declarations shared by the libflarepp translation units (not installed).
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/flarepp.h"

namespace flarepp {

constexpr int kNumSMs = 152;  // GB300: two dies of 76 SMs

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
    int64_t m_tile, n_mtiles;  // routes per encode CTA and route tiles per head
    int64_t m_pad;             // M rounded up for operand buffers
    // workspace layout (byte offsets from the workspace base, each 256-byte aligned)
    size_t off_pmax, off_psum, off_pacc;  // partials [BH][nchunk][M] f32 x2, [BH][nchunk][M][D] f32
    size_t off_q32, off_z32;              // Q, Z float32 [BH][M][D]
    size_t off_qop, off_zop;              // MMA operand copies of Q, Z (tensor-core path)
    size_t total;
};

// Fill `p` for `s`; returns FLAREPP_OK or the validation error for the shape itself.
flarepp_status make_plan(const flarepp_shape* s, Plan* p);

// ---- CUDA-core kernels (simt_kernels.cuh, instantiated in simt_f32.cu / simt_bf16.cu)
// Encode one call over all chunks: call 1 takes the seeds (element type of the inputs,
// [H][M][D]), call 2 takes Q32 from the workspace. Writes the chunk partials.
cudaError_t simt_encode_f32(const Plan& p, int call, const void* k, const void* v,
                            const void* seeds, float scale, char* ws, cudaStream_t st);
cudaError_t simt_encode_bf16(const Plan& p, int call, const void* k, const void* v,
                             const void* seeds, float scale, char* ws, cudaStream_t st);
// Decode (call 3) on CUDA cores: Y = SDPA(K, Q32, Z32).
cudaError_t simt_decode_f32(const Plan& p, const void* K, float scale, void* Y, char* ws,
                            cudaStream_t st);
cudaError_t simt_decode_bf16(const Plan& p, const void* K, float scale, void* Y, char* ws,
                             cudaStream_t st);

// ---- split-N combine (combine.cu)
// Stable log-sum-exp merge of the chunk partials into Q32 (call 1) or Z32 (call 2), plus
// the MMA operand copy when the tensor-core path consumes it.
cudaError_t combine(const Plan& p, int call, char* ws, cudaStream_t st);

}  // namespace flarepp
