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
// launch code (att::attend_launch) with the same work decomposition, but
// hands it one file-scope device array of fixed size for those partial
// results, and allocates nothing: no cudaMalloc, no cudaFree, no pool
// allocation.
//
// The array lives in every GPU that loads the library, until the process
// exits; each CUDA context has its own copy.  All calls within one context
// share it, so two calls whose kernels overlap on the GPU (different streams
// of one context) race on it; the caller must order such calls.  It keeps the
// last call's contents: nothing in it needs to start at zero, because every
// partial result a merge reads is written earlier in the same call, and the
// call clears the few arrival counters it keeps there itself
// (cudaMemsetAsync, which allocates nothing).
#include <mutex>

#include "internal.h"

using namespace att;

namespace {

// 32 MiB of split-KV partials: O (fp32, rows x d) and the row log-sum-exp.
constexpr size_t kStaticScratchBytes = 32ull << 20;
static __device__ __align__(256) unsigned char g_split_scratch[kStaticScratchBytes];

// In host code the array's name is only a host-side stand-in for the symbol:
// its device address has to be looked up (cudaGetSymbolAddress) with the
// right context current.  A module, and so the array, exists once per CUDA
// context, so the looked-up address is cached per context, keyed by the
// context's unique id (a context created after cudaDeviceReset, or a
// non-primary context, gets an id of its own and its own lookup).
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

constexpr int kCacheSlots = 64;
std::mutex g_setup_mutex;
unsigned long long g_ctx_id[kCacheSlots] = {0};
void* g_scratch_ptr[kCacheSlots] = {nullptr};
int g_next_slot = 0;

template <typename Fn>
Fn driver_fn(const char* name) {
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    return reinterpret_cast<Fn>(p);
  return nullptr;
}

// id of the calling thread's current context, or 0 if it cannot be told
unsigned long long current_context_id() {
  static CtxGetCurrentFn get_cur = driver_fn<CtxGetCurrentFn>("cuCtxGetCurrent");
  static CtxGetIdFn get_id = driver_fn<CtxGetIdFn>("cuCtxGetId");
  CUcontext c = nullptr;
  unsigned long long id = 0;
  if (!get_cur || !get_id || get_cur(&c) != CUDA_SUCCESS || c == nullptr || get_id(c, &id) != CUDA_SUCCESS)
    return 0;
  return id + 1;   // 0 stays "unknown"
}

// Device address of g_split_scratch in the current context (set-up on the
// first call in each context; later calls find it in the cache).
attuner_status scratch_address(void** out) {
  const unsigned long long id = current_context_id();
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (id != 0)
    for (int i = 0; i < kCacheSlots; ++i)
      if (g_ctx_id[i] == id) {
        *out = g_scratch_ptr[i];
        return ATTUNER_OK;
      }
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_split_scratch);
  if (e != cudaSuccess || p == nullptr)
    return fail(ATTUNER_ERR_CUDA,
                std::string("cudaGetSymbolAddress(split scratch) failed: ") + cudaGetErrorString(e));
  if (id != 0) {   // an unknown context is looked up on every call instead
    g_ctx_id[g_next_slot] = id;
    g_scratch_ptr[g_next_slot] = p;
    g_next_slot = (g_next_slot + 1) % kCacheSlots;
  }
  *out = p;
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
  FixedScratch fx{nullptr, kStaticScratchBytes};
  if ((e = scratch_address(&fx.base)) != ATTUNER_OK) return e;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int launches = 0;
  e = attend_launch(ctx, plan, q, suffix_k, suffix_v, S, S_kv, out, lse_out, st, &fx, launches);
  ctx->last_launches = launches;
  return finish_call(ctx, e, st);
}
