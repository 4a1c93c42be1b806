// attend_static.cu - attuner_attend_static_scratch: the attention step of
// attuner_attend for callers that cannot allocate GPU memory.
//
// Some callers own every byte of the device themselves: a serving engine
// that reserves the whole GPU for its own allocator up front, or a host
// runtime that forbids other libraries from calling cudaMalloc (or any
// stream-ordered allocator) because an allocation may synchronise the device
// or fail at an arbitrary point of a request.  attuner_attend draws its
// split-KV partial results from a stream-ordered pool, so it allocates on
// first use and whenever a call needs more.  This entry point runs the same
// kernels with the same work decomposition but keeps those partial results
// in one file-scope device array of fixed size instead, and allocates
// nothing: no cudaMalloc, no cudaFree, no pool allocation, no host heap.
//
// The array lives in every GPU that loads the library, until the process
// exits.  All calls share it, so two calls whose kernels overlap on the GPU
// (different streams, or different contexts on the same device) race on it;
// the caller must order such calls.  It keeps the last call's contents:
// nothing in it needs to start at zero, because every partial result a merge
// reads is written earlier in the same call, and the call clears the few
// arrival counters it keeps there itself (cudaMemsetAsync, which allocates
// nothing).
#include <mutex>

#include "internal.h"

using namespace att;

namespace {

// 32 MiB of split-KV partials: O (fp32, rows x d) and the row log-sum-exp.
constexpr size_t kStaticScratchBytes = 32ull << 20;
static __device__ __align__(256) unsigned char g_split_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {nullptr};

// Device address of g_split_scratch on the current device.  In host code the
// array's name is only a host-side stand-in for the symbol, so the address
// is looked up once per device (with that device current) and cached.
attuner_status scratch_address(int device, void** out) {
  if (device < 0 || device >= kMaxDevices)
    return fail(ATTUNER_ERR_UNSUPPORTED, "attuner_attend_static_scratch: device ordinal >= 64");
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_scratch_ptr[device] == nullptr) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_split_scratch);
    if (e != cudaSuccess || p == nullptr)
      return fail(ATTUNER_ERR_CUDA, std::string("cudaGetSymbolAddress(split scratch) failed: ") +
                                        cudaGetErrorString(e));
    g_scratch_ptr[device] = p;
  }
  *out = g_scratch_ptr[device];
  return ATTUNER_OK;
}

}  // namespace

extern "C" attuner_status attuner_attend_static_scratch(attuner_ctx* ctx, const attuner_plan* plan,
                                                        const void* q, const void* suffix_k,
                                                        const void* suffix_v, int32_t S, int32_t S_kv,
                                                        void* out, float* lse_out, void* stream) {
  attuner_status e = check_common(ctx, plan, S, S_kv);
  if (e != ATTUNER_OK) return e;
  if ((e = set_device(ctx)) != ATTUNER_OK) return e;
  CHECK_ARG(q && suffix_k && suffix_v && out, "q, suffix_k, suffix_v and out must not be NULL");
  CHECK_ARG(aligned16(q) && aligned16(suffix_k) && aligned16(suffix_v) && aligned16(out),
            "q, suffix_k, suffix_v and out must be 16-byte aligned");
  const attuner_config& c = ctx->cfg;
  const int D = c.head_dim, Hq = c.n_q_heads, Hkv = c.n_kv_heads, G = Hq / Hkv;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  bool tc;
  if (ctx->opt_prefill == 1) tc = true;
  else if (ctx->opt_prefill == 2) tc = false;
  else tc = (S * G > kMmaRows);
  const int rows = tc ? kTcRows : kMmaRows;

  AttnParams ap{};   // on the stack: this entry point touches no heap
  if (tc) query_cluster_occupancy(ctx);
  if ((e = make_work(ctx, plan, S, S_kv, tc, ap.work)) != ATTUNER_OK) return e;
  bool need_combine = false;   // split partial results in global memory
  for (int r = 0; r < plan->n_req; ++r) need_combine |= (ap.work.nsplit[r] > 1);
  if (ap.work.cluster > 0) need_combine = false;
  const size_t pb = need_combine ? (size_t)ap.work.n_cta * rows * (D + 1) * 4 : 0;
  const size_t units = (size_t)plan->n_req * Hkv * ap.work.row_tiles;
  const size_t part_bytes = pb + ((need_combine && tc) ? units * 4 : 0);
  if (part_bytes > kStaticScratchBytes)
    return fail(ATTUNER_ERR_INVALID_ARG,
                "attuner_attend_static_scratch: this call needs " + std::to_string(part_bytes) +
                    " bytes of split-KV scratch, more than the fixed " +
                    std::to_string(kStaticScratchBytes) + " bytes; use attuner_attend");
  void* scratch = nullptr;
  if (need_combine && (e = scratch_address(c.device, &scratch)) != ATTUNER_OK) return e;

  if (tc) {
    const uint64_t dims[5] = {(uint64_t)D, (uint64_t)G, (uint64_t)Hkv, (uint64_t)S, (uint64_t)plan->n_req};
    const uint64_t strides[4] = {(uint64_t)D * 2, (uint64_t)G * D * 2, (uint64_t)Hq * D * 2,
                                 (uint64_t)S * Hq * D * 2};
    const uint32_t box[5] = {64, (uint32_t)G, 1, (uint32_t)(kTcTileRows / G), 1};
    if ((e = make_map(&ap.tm_q, q, 5, dims, strides, box, "q")) != ATTUNER_OK) return e;
  }
  {
    const uint64_t dims[4] = {(uint64_t)D, (uint64_t)Hkv, (uint64_t)S_kv, (uint64_t)plan->n_req};
    const uint64_t strides[3] = {(uint64_t)D * 2, (uint64_t)Hkv * D * 2, (uint64_t)S_kv * Hkv * D * 2};
    const uint32_t box[4] = {64, 1, 64, 1};
    if ((e = make_map(&ap.tm_ksuf, suffix_k, 4, dims, strides, box, "suffix_k")) != ATTUNER_OK) return e;
    if ((e = make_map(&ap.tm_vsuf, suffix_v, 4, dims, strides, box, "suffix_v")) != ATTUNER_OK) return e;
  }
  if (tc && ap.work.cluster > 0 &&
      (e = make_out_map(&ap.tm_out, out, D, Hq, G, S, plan->n_req, ap.work.cluster)) != ATTUNER_OK)
    return e;
  ap.tm_kpool = ctx->tm_kpool;
  ap.tm_vpool = ctx->tm_vpool;
  ap.plan = plan_dev(plan);
  ap.q = static_cast<const __nv_bfloat16*>(q);
  ap.out = static_cast<__nv_bfloat16*>(out);
  ap.lse_out = lse_out;
  ap.S = S;
  ap.S_kv = S_kv;
  ap.Hq = Hq;
  ap.Hkv = Hkv;
  ap.G = G;
  ap.scale_log2 = (float)(1.4426950408889634 / sqrt((double)D));
  ap.status = ctx->d_status;
  ap.wait_limit = ctx->wait_limit;
  ap.inject_stuck = ctx->inject_stuck;
  cudaError_t ce = cudaSuccess;
  if (need_combine) {
    ap.part_o = static_cast<float*>(scratch);
    ap.part_lse = static_cast<float*>(scratch) + (size_t)ap.work.n_cta * rows * D;
    if (tc) {   // arrival counters of the in-kernel split merge
      ap.unit_cnt = reinterpret_cast<int*>(static_cast<char*>(scratch) + pb);
      ce = cudaMemsetAsync(ap.unit_cnt, 0, units * 4, st);
    }
  }
  int launches = 0;
  if (ce == cudaSuccess) ce = tc ? launch_attn_tc(ap, D, st) : launch_attn_mma(ap, D, st);
  if (ce == cudaSuccess) ++launches;
  if (ce == cudaSuccess && need_combine && !tc) {
    CombineParams cp{};
    cp.work = ap.work;
    cp.part_o = ap.part_o;
    cp.part_lse = ap.part_lse;
    cp.out = ap.out;
    cp.lse_out = lse_out;
    cp.S = S;
    cp.Hq = Hq;
    cp.Hkv = Hkv;
    cp.G = G;
    cp.D = D;
    cp.rows_per_tile = rows;
    ce = launch_combine(cp, st);
    if (ce == cudaSuccess) ++launches;
  }
  ctx->last_launches = launches;
  if (ce != cudaSuccess) return fail(ATTUNER_ERR_CUDA, std::string("attention launch failed: ") + cudaGetErrorString(ce));
  return finish_call(ctx, ATTUNER_OK, st);
}
