// kernels.h - launch parameters and host-side launchers of libattuner's
// kernels (internal to the library; the public boundary is attuner.h).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace att {

// K1: LoRA down-projection u = s * (A x) (bf16, zero-padded to 64 columns),
// B zero-padded to 64 columns, and the RoPE cos/sin table of every query row.
struct PrepParams {
  const __nv_bfloat16* x;        // [M, hidden]
  const __nv_bfloat16* lora_a;   // [r, hidden] or nullptr
  const __nv_bfloat16* lora_b;   // [d_q, r] or nullptr
  __nv_bfloat16* u_pad;          // [M, 64]
  __nv_bfloat16* b_pad;          // [d_q, 64]
  float2* rope;                  // [M, D/2] (cos, sin)
  const int32_t* t_art;          // [n_req]
  int32_t M, hidden, r, d_q, D, S, S_kv;
  float s;
  double inv_freq[64];           // theta^(-2j/D), j < D/2 (computed on the host in double)
};

// K1b: Q = RoPE(RMSNorm([x | u] [W_q | B]^T) * w)  (tcgen05 GEMM + epilogue)
struct QprojParams {
  CUtensorMap tm_x;    // x [M, hidden], box 64 x 128, SW128
  CUtensorMap tm_w;    // W_q [d_q, hidden], box 64 x D, SW128
  CUtensorMap tm_u;    // u_pad [M, 64], box 64 x 128
  CUtensorMap tm_b;    // b_pad [d_q, 64], box 64 x D
  __nv_bfloat16* q_out;            // [M, Hq, D]
  const __nv_bfloat16* qnorm_w;    // [D]
  const float2* rope;              // [M, D/2]
  int32_t M, hidden, Hq, lora_ksteps;
  float eps;
  int* status;
  long long wait_limit;
};

// K2 / K3: attention over assembled artifact blocks + suffix KV.
struct AttnParams {
  CUtensorMap tm_q;      // q [n_req, S, Hq, D] viewed 5-D (D, G, Hkv, S, n_req)   (K2 only)
  CUtensorMap tm_kpool;  // pool K viewed 2-D (D, pool_blocks*Hkv*64), box 64 x 64
  CUtensorMap tm_vpool;
  CUtensorMap tm_ksuf;   // suffix K viewed 4-D (D, Hkv, S_kv, n_req), box 64 x 1 x 64 x 1
  CUtensorMap tm_vsuf;
  PlanDev plan;
  WorkTable work;
  const __nv_bfloat16* q;        // (K3 reads Q directly)
  __nv_bfloat16* out;            // [n_req, S, Hq, D]
  float* lse_out;                // [n_req, S, Hq] or nullptr
  float* part_o;                 // [n_cta, rows_per_tile, D] (split chunks only)
  float* part_lse;               // [n_cta, rows_per_tile]
  int32_t S, S_kv, Hq, Hkv, G;
  float scale_log2;              // log2(e) / sqrt(D)
  int* status;
  long long wait_limit;
  int32_t inject_stuck;          // test hook: one role waits on a barrier nothing arrives at
};

struct CombineParams {
  WorkTable work;
  const float* part_o;
  const float* part_lse;
  __nv_bfloat16* out;
  float* lse_out;
  int32_t S, Hq, Hkv, G, D, rows_per_tile;
};

// Pool repack: caller K/V [L, Hkv, D] -> pool blocks [first + p/64][h][p%64][:]
cudaError_t launch_pool_write(const __nv_bfloat16* k, const __nv_bfloat16* v, __nv_bfloat16* kpool,
                              __nv_bfloat16* vpool, int L, int Hkv, int D, int first_block,
                              cudaStream_t st);
cudaError_t launch_prep(const PrepParams& p, cudaStream_t st);
cudaError_t launch_qproj(const QprojParams& p, int D, cudaStream_t st);
cudaError_t launch_attn_tc(const AttnParams& p, int D, cudaStream_t st);
cudaError_t launch_attn_mma(const AttnParams& p, int D, cudaStream_t st);
cudaError_t launch_combine(const CombineParams& p, cudaStream_t st);

// rows per CTA of each attention kernel
constexpr int kTcRows = 256;      // packed query rows per CTA of attn_tc (two tiles)
constexpr int kTcTileRows = 128;  // rows per query tile (one MMA M)
constexpr int kMmaRows = 16;
// largest split chunk (virtual blocks) the kernels' shared-memory block list holds
constexpr int kMaxChunkBlocks = 4096;

}  // namespace att
