// internal.h - host-side objects and helpers shared by the translation units
// that implement the C ABI (capi.cu and attend_static.cu).  Not part of the
// public boundary, which is include/attuner.h.
#pragma once

#include <mutex>
#include <string>
#include <unordered_set>
#include <utility>
#include <vector>

#include "kernels.h"

#define CUDA_TRY(call)                                                                        \
  do {                                                                                        \
    cudaError_t e_ = (call);                                                                  \
    if (e_ != cudaSuccess)                                                                    \
      return att::fail(ATTUNER_ERR_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

#define CHECK_ARG(cond, msg)                                       \
  do {                                                             \
    if (!(cond)) return att::fail(ATTUNER_ERR_INVALID_ARG, msg);   \
  } while (0)

using att::Artifact;

struct attuner_ctx {
  attuner_config cfg{};
  __nv_bfloat16* kpool = nullptr;
  __nv_bfloat16* vpool = nullptr;
  int32_t used_blocks = 0;
  uint64_t pool_gen = 0;          // attuner_pool_reset calls so far (plans record it)
  std::vector<Artifact> arts;
  CUtensorMap tm_kpool{}, tm_vpool{};
  int* d_status = nullptr;
  cudaMemPool_t mempool = nullptr;
  int num_sms = 0;
  int opt_prefill = 0;
  int opt_split = 0;
  int opt_qproj_split = 0;   // 0: the projection's shape from its cost model
  int opt_qproj_rows = 0;
  int opt_merge = 0;
  int opt_share = 0;          // shared artifact reads of the warp-MMA kernel: 0 auto, 1 off, 2 on
  int opt_sync_check = 0;
  int tc_clusters[9] = {-1, -1, -1, -1, -1, -1, -1, -1, -1};   // co-resident clusters of n tcgen05 CTAs
  long long wait_limit = 1ll << 32;
  int inject_stuck = 0;
  int last_launches = 0;
  double inv_freq[64] = {};       // theta^(-2j/d), j < d/2
  // plan uploads: a pinned staging buffer and a stream of the context's own
  // that does not synchronise with other streams, so assembling a plan waits
  // for its own copy only, never for kernels already running
  cudaStream_t upload_stream = nullptr;
  void* staging = nullptr;
  size_t staging_cap = 0;
  // device buffers of freed plans, reused by the next assemblies (capacity,
  // pointer), and the plans not yet freed (detached when the context goes, so
  // a plan freed after its context frees its own buffer)
  std::mutex plan_mu;
  std::vector<std::pair<size_t, int32_t*>> plan_bufs;
  std::unordered_set<attuner_plan*> live_plans;
};

// An assembled plan: the host tables (att::PlanTables) and their device copy.
struct attuner_plan : att::PlanTables {
  attuner_ctx* ctx = nullptr;     // owner of d_buf's cache; null once the context is destroyed
  size_t d_cap = 0;               // bytes of d_buf
  int32_t device = 0;
  int32_t pool_blocks = 0;
  uint64_t pool_gen = 0;          // the context's pool generation at assembly
  size_t spans_at = 0;            // int32 offset of spans in d_buf
  int32_t* d_buf = nullptr;       // blk_off | blocks | t_art | o_rows | span_off | spans
  // keys rotated at assembly (attuner_plan_rotate_keys): [n_slots][Hkv][64][d]
  // bf16, then the slots' assembled positions; null until rotated
  void* k_rot = nullptr;
  CUtensorMap tm_krot{};
};

namespace att {

// record `msg` as this thread's last error and return `s`
attuner_status fail(attuner_status s, const std::string& msg);
// bf16 tensor map with zero fill out of bounds; swizzle_bytes 128 (default),
// 64, 32 or 0 (none)
attuner_status make_map(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                        const uint64_t* strides, const uint32_t* box, const char* what,
                        int swizzle_bytes = 128);
// the cluster-mode output map of the tcgen05 attention kernel (see AttnParams::tm_out)
attuner_status make_out_map(CUtensorMap* m, void* out, int D, int Hq, int G, int S, int n_req, int cluster);
attuner_status set_device(const attuner_ctx* ctx);
bool aligned16(const void* p);
PlanDev plan_dev(const attuner_plan* p);
attuner_status check_common(attuner_ctx* ctx, const attuner_plan* plan, int S, int S_kv);
// split-KV decomposition of one attention launch (tc: tcgen05 kernel, else warp-MMA kernel)
attuner_status make_work(const attuner_ctx* ctx, const attuner_plan* plan, int S, int S_kv, bool tc, WorkTable& w,
                         int kv_part = 0);
// fills ctx->tc_clusters on first use (queries the device)
void query_cluster_occupancy(attuner_ctx* ctx);
// A caller-provided device region for the split-KV partial results of one
// attention launch, used instead of an allocation from the context's pool.
struct FixedScratch {
  void* base;   // device address, 256-byte aligned
  size_t cap;   // bytes
};
// The attention step of one call (attention and split-KV merge): work decomposition, tensor
// maps, split-KV scratch and the kernel launches on `st`.  With `fixed` null
// the scratch comes from the context's stream-ordered pool; otherwise from
// `fixed`, and a call needing more than fixed->cap bytes fails with
// INVALID_ARG before anything is launched.  Adds the kernels launched to
// `launches`.
// What a launch reads besides the plain read: which slots (kv_part as in
// SplitPolicy) and the softmax temperature of the logits.
struct AttendVariant {
  int kv_part = 0;
  float temperature = 1.f;
};
attuner_status attend_launch(attuner_ctx* ctx, const attuner_plan* plan, const void* q, const void* suffix_k,
                             const void* suffix_v, int32_t S, int32_t S_kv, void* out, float* lse_out,
                             cudaStream_t st, const FixedScratch* fixed, int& launches,
                             const AttendVariant& var = AttendVariant());
// the status a compute call returns: `e`, or with ATTUNER_OPT_SYNC_CHECK set
// and nothing failed on the host, the device status after `st` drains
attuner_status finish_call(attuner_ctx* ctx, attuner_status e, cudaStream_t st);

}  // namespace att
