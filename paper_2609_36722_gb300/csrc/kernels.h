// kernels.h - launch parameters and host-side launchers of libattuner's
// kernels (internal to the library; the public boundary is attuner.h).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace att {

// K1: the RoPE cos/sin table of every query row.
struct PrepParams {
  float2* rope;                  // [D/2, M] (cos, sin), pair-major
  PlanDev plan;                  // assembled positions of the online rows
  int32_t M, D, S, S_kv;
  double inv_freq[64];           // theta^(-2j/D), j < D/2 (computed on the host in double)
};

// K1b: Q = RoPE(RMSNorm(x W_q^T + s * bf16(x A^T) B^T) * w) as one tcgen05
// GEMM (A stacked under W_q: one MMA of N = D + r) with a fused epilogue.
// A CTA covers mr x 128 rows of one head and 1/ks of the K dimension (a
// cluster of ks CTAs per tile; see qproj.cu).
struct QprojParams {
  CUtensorMap tm_x;    // x [M, hidden], box 64 x 128, SW128
  CUtensorMap tm_w;    // W_q [d_q, hidden], box 64 x D, SW128
  CUtensorMap tm_a;    // A [r, hidden], box 64 x n_lora, SW128 (rows past r read as zeros)
  CUtensorMap tm_b;    // B [d_q, r], box 8 x D, no swizzle (columns past r read as zeros)
  CUtensorMap tm_w2;   // K/V mode: W_v [Hkv*D, hidden], box 64 x D, SW128
  __nv_bfloat16* q_out;            // Q mode: [M, Hq, D]; K/V mode: suffix K [n_req, S_kv, Hkv, D]
  __nv_bfloat16* out2;             // K/V mode: suffix V [n_req, S_kv, Hkv, D]
  const __nv_bfloat16* qnorm_w;    // [D] (q_norm, or k_norm in K/V mode)
  const float2* rope;              // [D/2, M] (cos, sin), pair-major
  int32_t M, hidden, Hq, r, n_lora;   // Hq: heads of the grid (2 Hkv in K/V mode)
  // K/V mode (kv = 1): grid heads [0, Hout) project K (W = tm_w, key norm and
  // RoPE), [Hout, 2 Hout) project V (W = tm_w2, stored as is).  Row m of the
  // GEMM is token m % S of request m / S, written to output token row
  // (m / S) * S_out + (S_out - S) + m % S (Q mode: S_out = S).
  int32_t kv, Hout, S, S_out;
  float s, eps;
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
  // cluster mode of K2 only: out viewed 4-D (D, Hq, S, n_req), box (D/cluster,
  // G, 256/G, 1), swizzle = the box row's bytes (32, 64 or 128)
  CUtensorMap tm_out;
  PlanDev plan;
  WorkTable work;
  const __nv_bfloat16* q;        // (K3 reads Q directly)
  __nv_bfloat16* out;            // [n_req, S, Hq, D]
  float* lse_out;                // [n_req, S, Hq] or nullptr
  float* part_o;                 // split chunks only: K3 [n_cta, 16, D] (shared reads: [n_part, Hkv, S G, D]);
                                 // K2 fp16 pieces (see attn_tc.cu)
  float* part_lse;               // [n_cta, rows_per_tile] (shared reads: [n_part, Hkv, S G])
  int* unit_cnt;                 // arrivals per (request, KV head, row tile); zero on entry
  int32_t S, S_kv, Hq, Hkv, G;
  float scale_log2;              // log2(e) / (sqrt(D) * temperature), temperature 1 but for APE's context part
  int* status;
  long long wait_limit;
  int32_t inject_stuck;          // test hook: one role waits on a barrier nothing arrives at
  // keys rotated at assembly (attuner_plan_rotate_keys): artifact slot s of
  // the plan (global slot index blk_off[req] + slot) reads its K from rows
  // (s * Hkv + kv head) * 64 of tm_kslot instead of the pool; V from the pool
  CUtensorMap tm_kslot;
  int32_t k_by_slot;
  int32_t kv_part;               // slots read: 0 all, 1 the plan's (artifacts), 2 the final online span
};


// Pool repack: caller K/V [L, Hkv, D] -> pool blocks [first + p/64][h][p%64][:]
// Batched pool write from host memory: artifact i copies [L[i], Hkv, D] K/V
// from k[i], v[i] (pinned host memory, read by the kernel over the CPU-GPU
// link) into pool blocks first[i] ...
struct HostBatch {
  const uint4* k[ATTUNER_MAX_HOST_BATCH];
  const uint4* v[ATTUNER_MAX_HOST_BATCH];
  long long chunk_end[ATTUNER_MAX_HOST_BATCH];   // inclusive prefix sums of L[i] * Hkv * D / 8
  int32_t L[ATTUNER_MAX_HOST_BATCH];
  int32_t first[ATTUNER_MAX_HOST_BATCH];
  int32_t n, Hkv, D;
};
// Keys rotated at assembly (App. C.2, EPIC paragraph): for every artifact
// slot s of a plan (entry blocks[s] > 0: pool block, valid tokens), token t
// of the slot is rotated at assembled position slot_pos[s] + t and written
// to krot[s][h][t][:] for every KV head h; rows t >= valid are zeroed.
// Online slots are skipped.
struct RotateParams {
  const uint4* kpool;            // [pool_blocks][Hkv][64][D] bf16, keys stored before RoPE
  uint4* krot;                   // [n_slots][Hkv][64][D] bf16
  const int32_t* blocks;         // [n_slots] the plan's slot entries
  const int32_t* slot_pos;       // [n_slots] assembled position of each slot's first token
  int32_t n_slots, Hkv, D, pool_blocks;
  int* status;
  double inv_freq[64];           // theta^(-2j/D), j < D/2
};
cudaError_t launch_rotate_keys(const RotateParams& p, cudaStream_t st);

// APE's calibrated combination (App. C.2, APE paragraph) of the context part
// (attention over the artifacts, logits divided by the temperature) and the
// online part (causal attention over the suffix), row by row:
//   w_c : w_o = exp(scale * lse_ctx) : exp(lse_on), out = w_c o_ctx + w_o o_on
//   (normalised), lse = log(exp(scale * lse_ctx) + exp(lse_on)).
// A request without artifacts (t_art 0) takes the online part alone.
struct ApeParams {
  const __nv_bfloat16* o_ctx;    // [n_req, S, Hq, D]
  const float* lse_ctx;          // [n_req, S, Hq]
  const __nv_bfloat16* o_on;
  const float* lse_on;
  __nv_bfloat16* out;
  float* lse_out;                // or nullptr
  const int32_t* t_art;          // [n_req]
  int32_t n_req, S, Hq, D;
  float scale;
};
cudaError_t launch_ape_combine(const ApeParams& p, cudaStream_t st);

cudaError_t launch_pool_write_host(const HostBatch& b, __nv_bfloat16* kpool, __nv_bfloat16* vpool,
                                   int num_sms, cudaStream_t st);
cudaError_t launch_pool_write(const __nv_bfloat16* k, const __nv_bfloat16* v, __nv_bfloat16* kpool,
                              __nv_bfloat16* vpool, int L, int Hkv, int D, int first_block,
                              cudaStream_t st);
cudaError_t launch_prep(const PrepParams& p, cudaStream_t st);
// Launch with mr accumulators of 128 rows per CTA and ks K slices per tile
// (qproj_shape_supported in plan.h lists the shapes).
cudaError_t launch_qproj(const QprojParams& p, int D, int mr, int ks, cudaStream_t st);
// Launch with programmatic stream serialization (the kernel may start while
// the previous kernel of the stream finishes; see grid_dep_wait) and, when
// cluster > 0, thread-block clusters of that many CTAs along x.
template <typename... Args>
cudaError_t launch_pdl(void (*kernel)(Args...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       int cluster, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  int n = 0;
  attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[n].val.programmaticStreamSerializationAllowed = 1;
  ++n;
  if (cluster > 0) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// how many clusters of `ns` tcgen05 attention CTAs fit on the current device at once
int attn_tc_max_clusters(int D, int ns);
cudaError_t launch_attn_tc(const AttnParams& p, int D, cudaStream_t st);
cudaError_t launch_attn_mma(const AttnParams& p, int D, cudaStream_t st);

}  // namespace att
