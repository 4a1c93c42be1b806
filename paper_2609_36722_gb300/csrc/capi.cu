// capi.cu - the C ABI of libattuner (declared in include/attuner.h):
// context and paged pool, artifact registration (bump allocation in
// registration order), request assembly into block tables and index maps,
// tensor-map encoding, split-KV work decomposition and kernel dispatch.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "internal.h"

using namespace att;

// ---------------------------------------------------------------------------
// errors
// ---------------------------------------------------------------------------
static thread_local std::string g_err;

attuner_status att::fail(attuner_status s, const std::string& msg) {
  g_err = msg;
  return s;
}

// ---------------------------------------------------------------------------
// driver entry point for tensor maps (no link-time dependency on libcuda)
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// bf16 tensor map, 128-byte swizzle (or none), zero fill out of bounds.
// dims[0] is the innermost (contiguous) dimension; strides[i] is the byte
// stride of dims[i+1].
attuner_status att::make_map(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                               const uint64_t* strides, const uint32_t* box, const char* what,
                               int swizzle_bytes) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return fail(ATTUNER_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  if ((reinterpret_cast<uintptr_t>(base) & 15) != 0)
    return fail(ATTUNER_ERR_INVALID_ARG, std::string(what) + ": base address must be 16-byte aligned");
  cuuint64_t d[5];
  cuuint64_t s[4];
  cuuint32_t b[5], e[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    b[i] = box[i];
    e[i] = 1;
    if (i + 1 < rank) s[i] = strides[i];
  }
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(base), d, s, b, e,
                  CU_TENSOR_MAP_INTERLEAVE_NONE,
                  swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                  : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                  : swizzle_bytes == 32 ? CU_TENSOR_MAP_SWIZZLE_32B
                                        : CU_TENSOR_MAP_SWIZZLE_NONE,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return fail(ATTUNER_ERR_CUDA, std::string("cuTensorMapEncodeTiled failed for ") + what +
                                      " (CUresult " + std::to_string((int)r) + ")");
  return ATTUNER_OK;
}

attuner_status att::make_out_map(CUtensorMap* m, void* out, int D, int Hq, int G, int S, int n_req,
                                 int cluster) {
  const int cw = D / cluster;   // columns one CTA writes: one box row of cw * 2 bytes
  const uint64_t dims[4] = {(uint64_t)D, (uint64_t)Hq, (uint64_t)S, (uint64_t)n_req};
  const uint64_t strides[3] = {(uint64_t)D * 2, (uint64_t)Hq * D * 2, (uint64_t)S * Hq * D * 2};
  const uint32_t box[4] = {(uint32_t)cw, (uint32_t)G, (uint32_t)(kTcRows / G), 1};
  return make_map(m, out, 4, dims, strides, box, "out", cw * 2);
}

attuner_status att::set_device(const attuner_ctx* ctx) {
  int cur = -1;
  CUDA_TRY(cudaGetDevice(&cur));
  if (cur != ctx->cfg.device) CUDA_TRY(cudaSetDevice(ctx->cfg.device));
  return ATTUNER_OK;
}

bool att::aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// stream-ordered scratch of one call
struct Scratch {
  attuner_ctx* ctx;
  cudaStream_t st;
  void* base = nullptr;
  size_t used = 0, cap = 0;
  size_t take(size_t bytes) {
    size_t off = used;
    used += (bytes + 255) & ~size_t(255);
    return off;
  }
};

// ---------------------------------------------------------------------------
// context
// ---------------------------------------------------------------------------
extern "C" attuner_status attuner_create(const attuner_config* cfg, attuner_ctx** out) {
  CHECK_ARG(cfg != nullptr && out != nullptr, "attuner_create: cfg and out must not be NULL");
  *out = nullptr;
  CHECK_ARG(cfg->head_dim == 64 || cfg->head_dim == 128, "head_dim must be 64 or 128");
  CHECK_ARG(cfg->n_kv_heads >= 1 && cfg->n_q_heads >= 1 && cfg->n_q_heads % cfg->n_kv_heads == 0,
            "n_q_heads must be a positive multiple of n_kv_heads");
  const int G = cfg->n_q_heads / cfg->n_kv_heads;
  CHECK_ARG(G == 1 || G == 2 || G == 4 || G == 8, "group size n_q_heads / n_kv_heads must be 1, 2, 4 or 8");
  CHECK_ARG(cfg->hidden >= 64 && cfg->hidden % 64 == 0, "hidden must be a positive multiple of 64");
  CHECK_ARG(cfg->block_tokens == ATTUNER_BLOCK_TOKENS, "block_tokens must be 64");
  CHECK_ARG(cfg->pool_blocks >= 1, "pool_blocks must be >= 1");
  CHECK_ARG((long long)cfg->pool_blocks * cfg->n_kv_heads * 64 < (1ll << 31),
            "pool too large: pool_blocks * n_kv_heads * 64 must be < 2^31");
  CHECK_ARG(cfg->pool_blocks < (1 << 24), "pool_blocks must be < 2^24");
  CHECK_ARG(cfg->rope_theta > 1.0f && cfg->rms_eps >= 0.0f, "rope_theta must be > 1 and rms_eps >= 0");
  int ndev = 0;
  CUDA_TRY(cudaGetDeviceCount(&ndev));
  CHECK_ARG(cfg->device >= 0 && cfg->device < ndev, "device ordinal out of range");

  attuner_ctx* ctx = new attuner_ctx();
  ctx->cfg = *cfg;
  attuner_status st = set_device(ctx);
  if (st != ATTUNER_OK) { delete ctx; return st; }
  const size_t pool_bytes = (size_t)cfg->pool_blocks * cfg->n_kv_heads * 64 * cfg->head_dim * 2;
  cudaError_t e1 = cudaMalloc(&ctx->kpool, pool_bytes);
  cudaError_t e2 = (e1 == cudaSuccess) ? cudaMalloc(&ctx->vpool, pool_bytes) : e1;
  cudaError_t e3 = (e2 == cudaSuccess) ? cudaMalloc(&ctx->d_status, sizeof(int)) : e2;
  if (e3 != cudaSuccess) {
    attuner_destroy(ctx);
    cudaGetLastError();
    return fail(ATTUNER_ERR_OOM, std::string("pool allocation failed: ") + cudaGetErrorString(e3));
  }
  if (cudaMemset(ctx->kpool, 0, pool_bytes) != cudaSuccess || cudaMemset(ctx->vpool, 0, pool_bytes) != cudaSuccess ||
      cudaMemset(ctx->d_status, 0, sizeof(int)) != cudaSuccess ||
      cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, cfg->device) != cudaSuccess) {
    attuner_destroy(ctx);
    return fail(ATTUNER_ERR_CUDA, "context initialisation failed");
  }
  cudaMemPoolProps props{};
  props.allocType = cudaMemAllocationTypePinned;
  props.location.type = cudaMemLocationTypeDevice;
  props.location.id = cfg->device;
  if (cudaMemPoolCreate(&ctx->mempool, &props) != cudaSuccess) {
    attuner_destroy(ctx);
    return fail(ATTUNER_ERR_CUDA, "cudaMemPoolCreate failed");
  }
  uint64_t thresh = ~0ull;
  cudaMemPoolSetAttribute(ctx->mempool, cudaMemPoolAttrReleaseThreshold, &thresh);
  if (cudaStreamCreateWithFlags(&ctx->upload_stream, cudaStreamNonBlocking) != cudaSuccess) {
    attuner_destroy(ctx);
    return fail(ATTUNER_ERR_CUDA, "cudaStreamCreateWithFlags failed");
  }
  for (int j = 0; j < cfg->head_dim / 2; ++j)
    ctx->inv_freq[j] = std::pow((double)cfg->rope_theta, -2.0 * j / (double)cfg->head_dim);

  const uint64_t D = cfg->head_dim;
  const uint64_t rows = (uint64_t)cfg->pool_blocks * cfg->n_kv_heads * 64;
  const uint64_t dims[2] = {D, rows};
  const uint64_t strides[1] = {D * 2};
  const uint32_t box[2] = {64, 64};
  st = make_map(&ctx->tm_kpool, ctx->kpool, 2, dims, strides, box, "K pool");
  if (st == ATTUNER_OK) st = make_map(&ctx->tm_vpool, ctx->vpool, 2, dims, strides, box, "V pool");
  if (st != ATTUNER_OK) {
    attuner_destroy(ctx);
    return st;
  }
  *out = ctx;
  return ATTUNER_OK;
}

extern "C" attuner_status attuner_destroy(attuner_ctx* ctx) {
  if (!ctx) return ATTUNER_OK;
  set_device(ctx);
  if (ctx->kpool) cudaFree(ctx->kpool);
  if (ctx->vpool) cudaFree(ctx->vpool);
  if (ctx->d_status) cudaFree(ctx->d_status);
  if (ctx->mempool) cudaMemPoolDestroy(ctx->mempool);
  if (ctx->upload_stream) cudaStreamDestroy(ctx->upload_stream);
  if (ctx->staging) cudaFreeHost(ctx->staging);
  {
    std::lock_guard<std::mutex> lk(ctx->plan_mu);
    for (attuner_plan* p : ctx->live_plans) p->ctx = nullptr;
    for (auto& b : ctx->plan_bufs) cudaFree(b.second);
  }
  delete ctx;
  return ATTUNER_OK;
}

extern "C" attuner_status attuner_register_artifact(attuner_ctx* ctx, const void* k, const void* v,
                                                    int32_t L, void* stream, int32_t* artifact_id_out) {
  CHECK_ARG(ctx != nullptr, "ctx must not be NULL");
  CHECK_ARG(k != nullptr && v != nullptr, "k and v must not be NULL");
  CHECK_ARG(L > 0 && L < (1 << 30), "artifact length L must be in [1, 2^30)");
  CHECK_ARG(aligned16(k) && aligned16(v), "k and v must be 16-byte aligned");
  const int nb = (L + 63) / 64;
  if ((long long)ctx->used_blocks + nb > ctx->cfg.pool_blocks)
    return fail(ATTUNER_ERR_OOM, "artifact pool is full: " + std::to_string(ctx->used_blocks) + " of " +
                                     std::to_string(ctx->cfg.pool_blocks) + " blocks used, " +
                                     std::to_string(nb) + " more needed");
  attuner_status s = set_device(ctx);
  if (s != ATTUNER_OK) return s;
  CUDA_TRY(launch_pool_write(static_cast<const __nv_bfloat16*>(k), static_cast<const __nv_bfloat16*>(v),
                             ctx->kpool, ctx->vpool, L, ctx->cfg.n_kv_heads, ctx->cfg.head_dim,
                             ctx->used_blocks, static_cast<cudaStream_t>(stream)));
  ctx->arts.push_back(Artifact{ctx->used_blocks, L, nb});
  ctx->used_blocks += nb;
  if (artifact_id_out) *artifact_id_out = (int32_t)ctx->arts.size() - 1;
  ctx->last_launches = 1;
  return ATTUNER_OK;
}

extern "C" attuner_status attuner_register_artifacts_host(attuner_ctx* ctx, int32_t n, const void* const* k_host,
                                                          const void* const* v_host, const int32_t* L,
                                                          void* stream, int32_t* ids_out) {
  CHECK_ARG(ctx != nullptr, "ctx must not be NULL");
  CHECK_ARG(n >= 1 && n <= ATTUNER_MAX_HOST_BATCH,
            "n must be in [1, " + std::to_string(ATTUNER_MAX_HOST_BATCH) + "]");
  CHECK_ARG(k_host != nullptr && v_host != nullptr && L != nullptr, "k_host, v_host and L must not be NULL");
  attuner_status s = set_device(ctx);
  if (s != ATTUNER_OK) return s;
  HostBatch* b = new HostBatch();
  auto done = [&](attuner_status st) { delete b; return st; };
  const int Hkv = ctx->cfg.n_kv_heads, D = ctx->cfg.head_dim;
  long long blocks = 0, chunks = 0;
  for (int i = 0; i < n; ++i) {
    if (L[i] <= 0 || L[i] >= (1 << 30))
      return done(fail(ATTUNER_ERR_INVALID_ARG, "artifact length L must be in [1, 2^30)"));
    if (!k_host[i] || !v_host[i] || !aligned16(k_host[i]) || !aligned16(v_host[i]))
      return done(fail(ATTUNER_ERR_INVALID_ARG, "k_host and v_host must be non-NULL and 16-byte aligned"));
    for (const void* ptr : {k_host[i], v_host[i]}) {
      cudaPointerAttributes at{};
      if (cudaPointerGetAttributes(&at, ptr) != cudaSuccess || at.type != cudaMemoryTypeHost) {
        cudaGetLastError();
        return done(fail(ATTUNER_ERR_INVALID_ARG, "k_host and v_host must be pinned host memory"));
      }
    }
    b->k[i] = static_cast<const uint4*>(k_host[i]);
    b->v[i] = static_cast<const uint4*>(v_host[i]);
    b->first[i] = ctx->used_blocks + (int)blocks;
    b->L[i] = L[i];
    blocks += (L[i] + 63) / 64;
    chunks += (long long)L[i] * Hkv * (D / 8);
    b->chunk_end[i] = chunks;
  }
  if (ctx->used_blocks + blocks > ctx->cfg.pool_blocks)
    return done(fail(ATTUNER_ERR_OOM, "artifact pool is full: " + std::to_string(ctx->used_blocks) + " of " +
                                          std::to_string(ctx->cfg.pool_blocks) + " blocks used, " +
                                          std::to_string(blocks) + " more needed"));
  b->n = n;
  b->Hkv = Hkv;
  b->D = D;
  const cudaError_t ce = launch_pool_write_host(*b, ctx->kpool, ctx->vpool, ctx->num_sms,
                                                static_cast<cudaStream_t>(stream));
  if (ce != cudaSuccess)
    return done(fail(ATTUNER_ERR_CUDA, std::string("pool write launch failed: ") + cudaGetErrorString(ce)));
  for (int i = 0; i < n; ++i) {
    ctx->arts.push_back(Artifact{b->first[i], L[i], (L[i] + 63) / 64});
    if (ids_out) ids_out[i] = (int32_t)ctx->arts.size() - 1;
  }
  ctx->used_blocks += (int32_t)blocks;
  ctx->last_launches = 1;
  return done(ATTUNER_OK);
}

extern "C" attuner_status attuner_pool_reset(attuner_ctx* ctx) {
  CHECK_ARG(ctx != nullptr, "ctx must not be NULL");
  ctx->arts.clear();
  ctx->used_blocks = 0;
  ++ctx->pool_gen;
  ctx->last_launches = 0;
  return ATTUNER_OK;
}

// ---------------------------------------------------------------------------
// plans
// ---------------------------------------------------------------------------
// Plans of both entry points: items >= 0 are artifact ids, items < 0 (layouts
// only) online spans of -item rows, in prompt order.
static attuner_status assemble_impl(attuner_ctx* ctx, const int32_t* ids, const int32_t* offs, int32_t n_req,
                                    bool layout, attuner_plan** out) {
  CHECK_ARG(ctx != nullptr && out != nullptr, "ctx and out must not be NULL");
  *out = nullptr;
  attuner_plan* p = new attuner_plan();
  std::string err;
  const attuner_status bs = build_plan_tables(ctx->arts, ids, offs, n_req, layout, *p, err);
  if (bs != ATTUNER_OK) {
    delete p;
    return fail(bs, err);
  }
  p->device = ctx->cfg.device;
  p->pool_blocks = ctx->cfg.pool_blocks;
  p->pool_gen = ctx->pool_gen;
  attuner_status s = set_device(ctx);
  if (s != ATTUNER_OK) { delete p; return s; }
  // the device image: blk_off | blocks | t_art | o_rows | span_off | req_art_off | ref_nblk |
  // dist_off | dist_src | dist_nb | dref_req | dref_j | dref_nref | (16-byte aligned) spans
  const std::vector<int32_t>* parts[] = {&p->blk_off, &p->blocks,   &p->t_art,   &p->o_rows,   &p->span_off,
                                         &p->req_art_off, &p->ref_nblk, &p->dist_off, &p->dist_src, &p->dist_nb,
                                         &p->dref_req, &p->dref_j, &p->dref_nref};
  size_t head = 0;
  for (const std::vector<int32_t>* v : parts) head += v->size();
  p->spans_at = (head + 3) & ~size_t(3);   // int4 spans start 16-byte aligned
  const size_t n_words = std::max<size_t>(p->spans_at + p->spans.size(), 1);
  const size_t bytes = n_words * sizeof(int32_t);
  if (ctx->staging_cap < bytes) {
    size_t cap = std::max<size_t>(ctx->staging_cap * 2, 1 << 16);
    while (cap < bytes) cap *= 2;
    void* st = nullptr;
    if (cudaMallocHost(&st, cap) != cudaSuccess) {
      cudaGetLastError();
      delete p;
      return fail(ATTUNER_ERR_OOM, "plan staging allocation failed");
    }
    if (ctx->staging) cudaFreeHost(ctx->staging);
    ctx->staging = st;
    ctx->staging_cap = cap;
  }
  {
    int32_t* h = static_cast<int32_t*>(ctx->staging);
    size_t at = 0;
    for (const std::vector<int32_t>* v : parts) {
      if (!v->empty()) std::memcpy(h + at, v->data(), v->size() * sizeof(int32_t));
      at += v->size();
    }
    for (; at < p->spans_at; ++at) h[at] = 0;
    if (!p->spans.empty()) std::memcpy(h + at, p->spans.data(), p->spans.size() * sizeof(int32_t));
  }
  // a buffer of a freed plan when one is large enough (no allocation per assembly)
  p->ctx = ctx;
  {
    std::lock_guard<std::mutex> lk(ctx->plan_mu);
    size_t best = ctx->plan_bufs.size();
    for (size_t i = 0; i < ctx->plan_bufs.size(); ++i)
      if (ctx->plan_bufs[i].first >= bytes && (best == ctx->plan_bufs.size() || ctx->plan_bufs[i].first < ctx->plan_bufs[best].first))
        best = i;
    if (best < ctx->plan_bufs.size()) {
      p->d_cap = ctx->plan_bufs[best].first;
      p->d_buf = ctx->plan_bufs[best].second;
      ctx->plan_bufs.erase(ctx->plan_bufs.begin() + best);
    }
  }
  if (!p->d_buf) {
    size_t cap = 4096;
    while (cap < bytes) cap *= 2;
    if (cudaMalloc(&p->d_buf, cap) != cudaSuccess) {
      cudaGetLastError();
      delete p;
      return fail(ATTUNER_ERR_OOM, "plan allocation failed");
    }
    p->d_cap = cap;
  }
  if (cudaMemcpyAsync(p->d_buf, ctx->staging, bytes, cudaMemcpyHostToDevice, ctx->upload_stream) != cudaSuccess ||
      cudaStreamSynchronize(ctx->upload_stream) != cudaSuccess) {
    cudaGetLastError();
    cudaFree(p->d_buf);
    delete p;
    return fail(ATTUNER_ERR_CUDA, "plan upload failed");
  }
  {
    std::lock_guard<std::mutex> lk(ctx->plan_mu);
    ctx->live_plans.insert(p);
  }
  *out = p;
  return ATTUNER_OK;
}

extern "C" attuner_status attuner_assemble(attuner_ctx* ctx, const int32_t* ids, const int32_t* offs,
                                           int32_t n_req, attuner_plan** out) {
  return assemble_impl(ctx, ids, offs, n_req, false, out);
}

extern "C" attuner_status attuner_assemble_layout(attuner_ctx* ctx, const int32_t* items, const int32_t* offs,
                                                  int32_t n_req, attuner_plan** out) {
  return assemble_impl(ctx, items, offs, n_req, true, out);
}

extern "C" attuner_status attuner_plan_export(const attuner_plan* p, int32_t* block_table, int32_t* valid_len,
                                              int32_t* index_map, int32_t* token_art, int32_t* token_off,
                                              int64_t* sizes) {
  CHECK_ARG(p != nullptr && sizes != nullptr, "plan and sizes_inout must not be NULL");
  std::string err;
  const attuner_status s = export_plan_tables(*p, block_table, valid_len, index_map, token_art, token_off, sizes,
                                              err);
  return s == ATTUNER_OK ? s : fail(s, err);
}

extern "C" attuner_status attuner_plan_t_art(const attuner_plan* p, int32_t* t_art, int32_t n_req) {
  CHECK_ARG(p != nullptr && t_art != nullptr, "plan and t_art_host must not be NULL");
  CHECK_ARG(n_req == p->n_req, "n_req does not match the plan");
  for (int i = 0; i < n_req; ++i) t_art[i] = p->t_art[i];
  return ATTUNER_OK;
}

extern "C" attuner_status attuner_plan_free(attuner_plan* p) {
  if (!p) return ATTUNER_OK;
  // keep the buffer for the context's next assemblies (a few at most)
  constexpr size_t kCachedPlanBufs = 8;
  if (p->ctx) {
    std::lock_guard<std::mutex> lk(p->ctx->plan_mu);
    p->ctx->live_plans.erase(p);
    if (p->d_buf && p->ctx->plan_bufs.size() < kCachedPlanBufs) {
      p->ctx->plan_bufs.emplace_back(p->d_cap, p->d_buf);
      p->d_buf = nullptr;
    }
  }
  if (p->d_buf || p->k_rot) {
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != p->device) cudaSetDevice(p->device);
    if (p->d_buf) cudaFree(p->d_buf);
    if (p->k_rot) cudaFree(p->k_rot);
    if (cur != p->device && cur >= 0) cudaSetDevice(cur);
  }
  delete p;
  return ATTUNER_OK;
}

// ---------------------------------------------------------------------------
// keys rotated at assembly (App. C.2, EPIC paragraph)
// ---------------------------------------------------------------------------
extern "C" attuner_status attuner_plan_rotate_keys(attuner_ctx* ctx, attuner_plan* plan, void* stream) {
  CHECK_ARG(ctx != nullptr && plan != nullptr, "ctx and plan must not be NULL");
  CHECK_ARG(plan->ctx == ctx, "plan belongs to another context");
  CHECK_ARG(plan->pool_gen == ctx->pool_gen, "plan was assembled before the last attuner_pool_reset");
  if (plan->max_o_rows > 0)
    return fail(ATTUNER_ERR_UNSUPPORTED, "attuner_plan_rotate_keys: plans with online spans between artifacts");
  attuner_status e = set_device(ctx);
  if (e != ATTUNER_OK) return e;
  const attuner_config& c = ctx->cfg;
  const int D = c.head_dim, Hkv = c.n_kv_heads;
  const size_t n_slots = plan->blocks.size();
  if (n_slots == 0) return ATTUNER_OK;   // no artifact: nothing to rotate, the plain read is the same
  CHECK_ARG((long long)n_slots * Hkv * kBlockTokens < (1ll << 31), "plan too large to rotate (slots * Hkv * 64 >= 2^31)");
  // assembled position of each slot's first token: the request's artifact
  // tokens before it, in runtime order from position 0
  std::vector<int32_t> pos(n_slots, 0);
  for (int r = 0; r < plan->n_req; ++r) {
    int32_t at = 0;
    for (int b = plan->blk_off[r]; b < plan->blk_off[r + 1]; ++b) {
      pos[b] = at;
      at += plan->blocks[b] & 127;
    }
  }
  const size_t key_bytes = n_slots * Hkv * kBlockTokens * D * 2;
  if (plan->k_rot == nullptr) {
    if (cudaMalloc(&plan->k_rot, key_bytes + n_slots * 4) != cudaSuccess) {
      cudaGetLastError();
      plan->k_rot = nullptr;
      return fail(ATTUNER_ERR_OOM, "rotated-key allocation failed");
    }
    const uint64_t dims[2] = {(uint64_t)D, (uint64_t)n_slots * Hkv * kBlockTokens};
    const uint64_t strides[1] = {(uint64_t)D * 2};
    const uint32_t box[2] = {64, 64};
    if ((e = make_map(&plan->tm_krot, plan->k_rot, 2, dims, strides, box, "rotated keys")) != ATTUNER_OK) {
      cudaFree(plan->k_rot);
      plan->k_rot = nullptr;
      return e;
    }
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int32_t* d_pos = reinterpret_cast<int32_t*>(static_cast<char*>(plan->k_rot) + key_bytes);
  CUDA_TRY(cudaMemcpyAsync(d_pos, pos.data(), n_slots * 4, cudaMemcpyHostToDevice, st));
  RotateParams rp{};
  rp.kpool = reinterpret_cast<const uint4*>(ctx->kpool);
  rp.krot = reinterpret_cast<uint4*>(plan->k_rot);
  rp.blocks = plan_dev(plan).blocks;
  rp.slot_pos = d_pos;
  rp.n_slots = (int32_t)n_slots;
  rp.Hkv = Hkv;
  rp.D = D;
  rp.pool_blocks = c.pool_blocks;
  rp.status = ctx->d_status;
  for (int j = 0; j < D / 2; ++j) rp.inv_freq[j] = ctx->inv_freq[j];
  CUDA_TRY(launch_rotate_keys(rp, st));
  // the positions are read by the kernel from pageable host memory's copy:
  // keep `pos` alive until the copy has been made
  CUDA_TRY(cudaStreamSynchronize(st));
  ctx->last_launches = 1;
  return finish_call(ctx, ATTUNER_OK, st);
}

PlanDev att::plan_dev(const attuner_plan* p) {
  PlanDev d;
  d.blk_off = p->d_buf;
  d.blocks = p->d_buf + p->blk_off.size();
  d.t_art = p->d_buf + p->blk_off.size() + p->blocks.size();
  d.o_rows = d.t_art + p->t_art.size();
  d.span_off = d.o_rows + p->o_rows.size();
  d.req_art_off = d.span_off + p->span_off.size();
  d.ref_nblk = d.req_art_off + p->req_art_off.size();
  d.dist_off = d.ref_nblk + p->ref_nblk.size();
  d.dist_src = d.dist_off + p->dist_off.size();
  d.dist_nb = d.dist_src + p->dist_src.size();
  d.dref_req = d.dist_nb + p->dist_nb.size();
  d.dref_j = d.dref_req + p->dref_req.size();
  d.dref_nref = d.dref_j + p->dref_j.size();
  d.spans = reinterpret_cast<const int4*>(p->d_buf + p->spans_at);
  d.pool_blocks = p->pool_blocks;
  d.has_spans = p->max_o_rows > 0 ? 1 : 0;
  return d;
}

// ---------------------------------------------------------------------------
// Q projection
// ---------------------------------------------------------------------------
attuner_status att::check_common(attuner_ctx* ctx, const attuner_plan* plan, int S, int S_kv) {
  CHECK_ARG(ctx != nullptr && plan != nullptr, "ctx and plan must not be NULL");
  CHECK_ARG(plan->ctx == ctx, "plan belongs to another context");
  CHECK_ARG(plan->pool_gen == ctx->pool_gen, "plan was assembled before the last attuner_pool_reset");
  CHECK_ARG(S >= 1 && S_kv >= S, "need 1 <= S <= S_kv");
  CHECK_ARG((long long)plan->n_req * S * ctx->cfg.n_q_heads < (1ll << 31) && S_kv < (1 << 22),
            "n_req * S * n_q_heads must be < 2^31 and S_kv < 2^22");
  CHECK_ARG(S_kv >= plan->max_o_rows, "S_kv must cover the online rows of the plan's spans");
  return ATTUNER_OK;
}

// Launch shape of the projection kernel (choose_qproj_shape in plan.cpp):
// rows per CTA and K slices per tile, from the context's options and SM count.
static QpShape qproj_shape(const attuner_ctx* ctx, int heads, int M, int n_lora) {
  QpPolicy pol;
  pol.head_dim = ctx->cfg.head_dim;
  pol.hidden = ctx->cfg.hidden;
  pol.num_sms = ctx->num_sms;
  pol.opt_rows = ctx->opt_qproj_rows;
  pol.opt_split = ctx->opt_qproj_split;
  return choose_qproj_shape(pol, heads, M, n_lora);
}

static attuner_status q_project_impl(attuner_ctx* ctx, const attuner_plan* plan, const void* x, const void* w_q,
                                     const void* lora_a, const void* lora_b, int32_t r, float s,
                                     const void* q_norm_w, int32_t S, int32_t S_kv, void* q_out,
                                     cudaStream_t st, Scratch& sc, int& launches) {
  const attuner_config& c = ctx->cfg;
  CHECK_ARG(x && w_q && q_norm_w && q_out, "x, w_q, q_norm_w and q_out must not be NULL");
  CHECK_ARG(aligned16(x) && aligned16(w_q) && aligned16(q_out) && aligned16(q_norm_w),
            "x, w_q, q_norm_w and q_out must be 16-byte aligned");
  const bool lora = (r > 0 && lora_a != nullptr && lora_b != nullptr);
  CHECK_ARG(r >= 0 && r <= 64 && r % 8 == 0, "LoRA rank r must be 0 or a multiple of 8 up to 64");
  if (lora) CHECK_ARG(aligned16(lora_a) && aligned16(lora_b), "lora_a and lora_b must be 16-byte aligned");
  const int M = plan->n_req * S;
  const int D = c.head_dim, Hq = c.n_q_heads, dq = Hq * D;
  const int n_lora = lora ? ((r + 15) / 16) * 16 : 0;
  const QpShape shape = qproj_shape(ctx, Hq, M, n_lora);
  CHECK_ARG(shape.mr != 0, "ATTUNER_OPT_QPROJ_SPLIT_K / ATTUNER_OPT_QPROJ_ROWS leave no supported "
                           "projection shape for this head size, LoRA rank and hidden size");
  const size_t off_rope = sc.take((size_t)M * (D / 2) * 8);
  char* base = static_cast<char*>(sc.base);
  float2* rope = reinterpret_cast<float2*>(base + off_rope);

  PrepParams pp{};
  pp.rope = rope;
  pp.plan = plan_dev(plan);
  pp.M = M;
  pp.D = D;
  pp.S = S;
  pp.S_kv = S_kv;
  for (int j = 0; j < D / 2; ++j) pp.inv_freq[j] = ctx->inv_freq[j];
  CUDA_TRY(launch_prep(pp, st));
  ++launches;

  QprojParams qp{};
  attuner_status e;
  {
    const uint64_t dims[2] = {(uint64_t)c.hidden, (uint64_t)M};
    const uint64_t strides[1] = {(uint64_t)c.hidden * 2};
    const uint32_t box[2] = {64, 128};
    if ((e = make_map(&qp.tm_x, x, 2, dims, strides, box, "x")) != ATTUNER_OK) return e;
  }
  {
    const uint64_t dims[2] = {(uint64_t)c.hidden, (uint64_t)dq};
    const uint64_t strides[1] = {(uint64_t)c.hidden * 2};
    const uint32_t box[2] = {64, (uint32_t)D};
    if ((e = make_map(&qp.tm_w, w_q, 2, dims, strides, box, "w_q")) != ATTUNER_OK) return e;
  }
  if (lora) {
    const uint64_t dims[2] = {(uint64_t)c.hidden, (uint64_t)r};
    const uint64_t strides[1] = {(uint64_t)c.hidden * 2};
    const uint32_t box[2] = {64, (uint32_t)n_lora};
    if ((e = make_map(&qp.tm_a, lora_a, 2, dims, strides, box, "lora_a")) != ATTUNER_OK) return e;
    const uint64_t bdims[2] = {(uint64_t)r, (uint64_t)dq};
    const uint64_t bstrides[1] = {(uint64_t)r * 2};
    const uint32_t bbox[2] = {8, (uint32_t)D};
    if ((e = make_map(&qp.tm_b, lora_b, 2, bdims, bstrides, bbox, "lora_b", 0)) != ATTUNER_OK) return e;
  }
  qp.q_out = static_cast<__nv_bfloat16*>(q_out);
  qp.qnorm_w = static_cast<const __nv_bfloat16*>(q_norm_w);
  qp.rope = rope;
  qp.M = M;
  qp.hidden = c.hidden;
  qp.Hq = Hq;
  qp.kv = 0;
  qp.Hout = Hq;
  qp.S = S;
  qp.S_out = S;
  qp.r = lora ? r : 0;
  qp.n_lora = n_lora;
  qp.s = s;
  qp.eps = c.rms_eps;
  qp.status = ctx->d_status;
  qp.wait_limit = ctx->wait_limit;
  CUDA_TRY(launch_qproj(qp, D, shape.mr, shape.ks, st));
  ++launches;
  return ATTUNER_OK;
}

// The suffix tokens' own K and V: one launch of the Q-projection kernel in
// K/V mode (grid heads 0..Hkv-1 project K with the key norm and RoPE, Hkv..
// 2 Hkv-1 project V), after the prep kernel's RoPE table of the same positions.
static attuner_status kv_project_impl(attuner_ctx* ctx, const attuner_plan* plan, const void* x,
                                      const void* w_k, const void* w_v, const void* k_norm_w, int32_t S,
                                      int32_t S_kv, void* suffix_k, void* suffix_v, cudaStream_t st,
                                      Scratch& sc, int& launches) {
  const attuner_config& c = ctx->cfg;
  CHECK_ARG(x && w_k && w_v && k_norm_w && suffix_k && suffix_v,
            "x, w_k, w_v, k_norm_w, suffix_k and suffix_v must not be NULL");
  CHECK_ARG(aligned16(x) && aligned16(w_k) && aligned16(w_v) && aligned16(k_norm_w) && aligned16(suffix_k) &&
                aligned16(suffix_v),
            "x, w_k, w_v, k_norm_w, suffix_k and suffix_v must be 16-byte aligned");
  const int M = plan->n_req * S;
  const int D = c.head_dim, Hkv = c.n_kv_heads, dkv = Hkv * D;
  const size_t off_rope = sc.take((size_t)M * (D / 2) * 8);
  char* base = static_cast<char*>(sc.base);
  float2* rope = reinterpret_cast<float2*>(base + off_rope);

  PrepParams pp{};
  pp.rope = rope;
  pp.plan = plan_dev(plan);
  pp.M = M;
  pp.D = D;
  pp.S = S;
  pp.S_kv = S_kv;
  for (int j = 0; j < D / 2; ++j) pp.inv_freq[j] = ctx->inv_freq[j];
  CUDA_TRY(launch_prep(pp, st));
  ++launches;

  QprojParams qp{};
  attuner_status e;
  {
    const uint64_t dims[2] = {(uint64_t)c.hidden, (uint64_t)M};
    const uint64_t strides[1] = {(uint64_t)c.hidden * 2};
    const uint32_t box[2] = {64, 128};
    if ((e = make_map(&qp.tm_x, x, 2, dims, strides, box, "x")) != ATTUNER_OK) return e;
  }
  const QpShape shape = qproj_shape(ctx, 2 * Hkv, M, 0);
  CHECK_ARG(shape.mr != 0, "ATTUNER_OPT_QPROJ_SPLIT_K / ATTUNER_OPT_QPROJ_ROWS leave no supported "
                           "projection shape for this head size and hidden size");
  {
    const uint64_t dims[2] = {(uint64_t)c.hidden, (uint64_t)dkv};
    const uint64_t strides[1] = {(uint64_t)c.hidden * 2};
    const uint32_t box[2] = {64, (uint32_t)D};
    if ((e = make_map(&qp.tm_w, w_k, 2, dims, strides, box, "w_k")) != ATTUNER_OK) return e;
    if ((e = make_map(&qp.tm_w2, w_v, 2, dims, strides, box, "w_v")) != ATTUNER_OK) return e;
  }
  qp.q_out = static_cast<__nv_bfloat16*>(suffix_k);
  qp.out2 = static_cast<__nv_bfloat16*>(suffix_v);
  qp.qnorm_w = static_cast<const __nv_bfloat16*>(k_norm_w);
  qp.rope = rope;
  qp.M = M;
  qp.hidden = c.hidden;
  qp.Hq = 2 * Hkv;
  qp.kv = 1;
  qp.Hout = Hkv;
  qp.S = S;
  qp.S_out = S_kv;
  qp.r = 0;
  qp.n_lora = 0;
  qp.s = 0.f;
  qp.eps = c.rms_eps;
  qp.status = ctx->d_status;
  qp.wait_limit = ctx->wait_limit;
  CUDA_TRY(launch_qproj(qp, D, shape.mr, shape.ks, st));
  ++launches;
  return ATTUNER_OK;
}

static size_t q_project_scratch(const attuner_ctx* ctx, int M) {
  const int D = ctx->cfg.head_dim;
  auto al = [](size_t b) { return (b + 255) & ~size_t(255); };
  return al((size_t)M * (D / 2) * 8);
}

// ---------------------------------------------------------------------------
// attention
// ---------------------------------------------------------------------------
void att::query_cluster_occupancy(attuner_ctx* ctx) {
  if (ctx->tc_clusters[2] >= 0) return;
  for (int ns = 0; ns <= 8; ++ns)
    ctx->tc_clusters[ns] = (ns == 2 || ns == 4) ? attn_tc_max_clusters(ctx->cfg.head_dim, ns) : 0;
}

attuner_status att::make_work(const attuner_ctx* ctx, const attuner_plan* plan, int S, int S_kv, bool tc,
                              WorkTable& w, int kv_part) {
  SplitPolicy pol;
  pol.kv_part = kv_part;
  pol.n_q_heads = ctx->cfg.n_q_heads;
  pol.n_kv_heads = ctx->cfg.n_kv_heads;
  pol.num_sms = ctx->num_sms;
  pol.opt_split = ctx->opt_split;
  pol.opt_merge = ctx->opt_merge;
  pol.opt_share = ctx->opt_share;
  pol.k_by_slot = plan->k_rot != nullptr ? 1 : 0;
  for (int i = 0; i < 9; ++i) pol.tc_clusters[i] = ctx->tc_clusters[i];
  std::string err;
  const attuner_status s = split_work(pol, *plan, S, S_kv, tc, w, err);
  return s == ATTUNER_OK ? s : fail(s, err);
}

attuner_status att::attend_launch(attuner_ctx* ctx, const attuner_plan* plan, const void* q,
                                  const void* suffix_k, const void* suffix_v, int32_t S, int32_t S_kv,
                                  void* out, float* lse_out, cudaStream_t st, const FixedScratch* fixed,
                                  int& launches, const AttendVariant& var) {
  const attuner_config& c = ctx->cfg;
  CHECK_ARG(q && suffix_k && suffix_v && out, "q, suffix_k, suffix_v and out must not be NULL");
  CHECK_ARG(aligned16(q) && aligned16(suffix_k) && aligned16(suffix_v) && aligned16(out),
            "q, suffix_k, suffix_v and out must be 16-byte aligned");
  const int D = c.head_dim, Hq = c.n_q_heads, Hkv = c.n_kv_heads, G = Hq / Hkv;
  bool tc;
  if (ctx->opt_prefill == 1) tc = true;
  else if (ctx->opt_prefill == 2) tc = false;
  else tc = (S * G > kMmaRows);
  const int rows = tc ? kTcRows : kMmaRows;

  AttnParams ap{};   // on the stack: the launch itself touches no heap
  attuner_status e = ATTUNER_OK;
  if (tc) query_cluster_occupancy(ctx);
  if ((e = make_work(ctx, plan, S, S_kv, tc, ap.work, var.kv_part)) != ATTUNER_OK) return e;
  const WorkTable& w = ap.work;
  if (w.n_cta == 0) return ATTUNER_OK;   // no request has a slot of this part
  bool need_combine = w.share != 0;   // split partial results in global memory
  if (!w.share)
    for (int r = 0; r < plan->n_req; ++r) need_combine |= (w.nsplit[r] > 1);
  if (w.cluster > 0) need_combine = false;
  // partial O and LSE of every split CTA (shared reads: of every partial
  // record, the S G rows of one request) and one arrival counter per (request,
  // KV head, row tile), zeroed below: the last CTA of a row tile to arrive
  // merges its chunks, in either kernel
  const size_t records = w.share ? (size_t)w.n_part * Hkv : (size_t)w.n_cta;
  const size_t rec_rows = w.share ? (size_t)S * G : (size_t)rows;
  const size_t pb = need_combine ? records * rec_rows * (D + 1) * 4 : 0;
  const size_t units = (size_t)plan->n_req * Hkv * w.row_tiles;
  const size_t part_bytes = pb + (need_combine ? units * 4 : 0);
  if (fixed && part_bytes > fixed->cap)
    return fail(ATTUNER_ERR_INVALID_ARG,
                "this call needs " + std::to_string(part_bytes) + " bytes of split-KV scratch, more than the fixed " +
                    std::to_string(fixed->cap) + " bytes of attuner_attend_static_scratch; use attuner_attend");

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
  if (tc && w.cluster > 0 &&
      (e = make_out_map(&ap.tm_out, out, D, Hq, G, S, plan->n_req, w.cluster)) != ATTUNER_OK)
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
  ap.scale_log2 = (float)(1.4426950408889634 / (std::sqrt((double)D) * (double)var.temperature));
  ap.status = ctx->d_status;
  ap.wait_limit = ctx->wait_limit;
  ap.inject_stuck = ctx->inject_stuck;
  ap.kv_part = var.kv_part;
  if (plan->k_rot != nullptr) {
    ap.k_by_slot = 1;
    ap.tm_kslot = plan->tm_krot;
  }

  void* part = nullptr;
  cudaError_t ce = cudaSuccess;
  if (need_combine) {
    if (fixed) {
      part = fixed->base;
    } else if (cudaMallocFromPoolAsync(&part, part_bytes, ctx->mempool, st) != cudaSuccess) {
      cudaGetLastError();
      return fail(ATTUNER_ERR_OOM, "split-KV scratch allocation failed");
    }
    ap.part_o = static_cast<float*>(part);
    ap.part_lse = static_cast<float*>(part) + records * rec_rows * D;
    ap.unit_cnt = reinterpret_cast<int*>(static_cast<char*>(part) + pb);
    ce = cudaMemsetAsync(ap.unit_cnt, 0, units * 4, st);
  }
  if (ce == cudaSuccess) ce = tc ? launch_attn_tc(ap, D, st) : launch_attn_mma(ap, D, st);
  if (ce == cudaSuccess) ++launches;
  if (part && !fixed) cudaFreeAsync(part, st);
  if (ce != cudaSuccess) return fail(ATTUNER_ERR_CUDA, std::string("attention launch failed: ") + cudaGetErrorString(ce));
  return ATTUNER_OK;
}

extern "C" attuner_status attuner_q_project(attuner_ctx* ctx, const attuner_plan* plan, const void* x,
                                            const void* w_q, const void* lora_a, const void* lora_b, int32_t r,
                                            float s, const void* q_norm_w, int32_t S, int32_t S_kv, void* q_out,
                                            void* stream) {
  attuner_status e = check_common(ctx, plan, S, S_kv);
  if (e != ATTUNER_OK) return e;
  if ((e = set_device(ctx)) != ATTUNER_OK) return e;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  Scratch sc{ctx, st};
  sc.cap = q_project_scratch(ctx, plan->n_req * S);
  CUDA_TRY(cudaMallocFromPoolAsync(&sc.base, sc.cap, ctx->mempool, st));
  int launches = 0;
  e = q_project_impl(ctx, plan, x, w_q, lora_a, lora_b, r, s, q_norm_w, S, S_kv, q_out, st, sc, launches);
  cudaFreeAsync(sc.base, st);
  ctx->last_launches = launches;
  return finish_call(ctx, e, st);
}

extern "C" attuner_status attuner_kv_project(attuner_ctx* ctx, const attuner_plan* plan, const void* x,
                                             const void* w_k, const void* w_v, const void* k_norm_w, int32_t S,
                                             int32_t S_kv, void* suffix_k, void* suffix_v, void* stream) {
  attuner_status e = check_common(ctx, plan, S, S_kv);
  if (e != ATTUNER_OK) return e;
  if ((e = set_device(ctx)) != ATTUNER_OK) return e;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  Scratch sc{ctx, st};
  auto al = [](size_t b) { return (b + 255) & ~size_t(255); };
  sc.cap = al((size_t)plan->n_req * S * (ctx->cfg.head_dim / 2) * 8);
  CUDA_TRY(cudaMallocFromPoolAsync(&sc.base, sc.cap, ctx->mempool, st));
  int launches = 0;
  e = kv_project_impl(ctx, plan, x, w_k, w_v, k_norm_w, S, S_kv, suffix_k, suffix_v, st, sc, launches);
  cudaFreeAsync(sc.base, st);
  ctx->last_launches = launches;
  return finish_call(ctx, e, st);
}

extern "C" attuner_status attuner_attend(attuner_ctx* ctx, const attuner_plan* plan, const void* q,
                                         const void* suffix_k, const void* suffix_v, int32_t S, int32_t S_kv,
                                         void* out, float* lse_out, void* stream) {
  attuner_status e = check_common(ctx, plan, S, S_kv);
  if (e != ATTUNER_OK) return e;
  if ((e = set_device(ctx)) != ATTUNER_OK) return e;
  int launches = 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  e = attend_launch(ctx, plan, q, suffix_k, suffix_v, S, S_kv, out, lse_out, st, nullptr, launches);
  ctx->last_launches = launches;
  return finish_call(ctx, e, st);
}

extern "C" attuner_status attuner_query_attend(attuner_ctx* ctx, const attuner_plan* plan, const void* x,
                                               const void* w_q, const void* lora_a, const void* lora_b,
                                               int32_t r, float s, const void* q_norm_w, const void* suffix_k,
                                               const void* suffix_v, int32_t S, int32_t S_kv, void* out,
                                               float* lse_out, void* stream) {
  attuner_status e = check_common(ctx, plan, S, S_kv);
  if (e != ATTUNER_OK) return e;
  if ((e = set_device(ctx)) != ATTUNER_OK) return e;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int M = plan->n_req * S;
  const size_t q_bytes = ((size_t)M * ctx->cfg.n_q_heads * ctx->cfg.head_dim * 2 + 255) & ~size_t(255);
  Scratch sc{ctx, st};
  sc.cap = q_bytes + q_project_scratch(ctx, M);
  CUDA_TRY(cudaMallocFromPoolAsync(&sc.base, sc.cap, ctx->mempool, st));
  const size_t off_q = sc.take(q_bytes);
  void* q = static_cast<char*>(sc.base) + off_q;
  int launches = 0;
  e = q_project_impl(ctx, plan, x, w_q, lora_a, lora_b, r, s, q_norm_w, S, S_kv, q, st, sc, launches);
  if (e == ATTUNER_OK)
    e = attend_launch(ctx, plan, q, suffix_k, suffix_v, S, S_kv, out, lse_out, st, nullptr, launches);
  cudaFreeAsync(sc.base, st);
  ctx->last_launches = launches;
  return finish_call(ctx, e, st);
}

// The whole path with the step's new inputs and its output in host memory:
// the copies in, the projection and attention of attuner_query_attend, and
// the copies out, all enqueued on the caller's stream from one host call.
extern "C" attuner_status attuner_query_attend_host(attuner_ctx* ctx, const attuner_plan* plan, const void* x_host,
                                                    const void* w_q, const void* lora_a, const void* lora_b,
                                                    int32_t r, float s, const void* q_norm_w, const void* k_new_host,
                                                    const void* v_new_host, void* suffix_k, void* suffix_v, int32_t S,
                                                    int32_t S_kv, void* out_host, float* lse_host, void* stream) {
  attuner_status e = check_common(ctx, plan, S, S_kv);
  if (e != ATTUNER_OK) return e;
  CHECK_ARG(x_host != nullptr && out_host != nullptr && suffix_k != nullptr && suffix_v != nullptr,
            "x_host, out_host, suffix_k and suffix_v must not be NULL");
  CHECK_ARG((k_new_host == nullptr) == (v_new_host == nullptr),
            "k_new_host and v_new_host must both be given or both be NULL");
  if ((e = set_device(ctx)) != ATTUNER_OK) return e;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const attuner_config& c = ctx->cfg;
  const int M = plan->n_req * S;
  auto al = [](size_t b) { return (b + 255) & ~size_t(255); };
  const size_t x_bytes = (size_t)M * c.hidden * 2;
  const size_t o_bytes = (size_t)M * c.n_q_heads * c.head_dim * 2;
  const size_t l_bytes = lse_host ? (size_t)M * c.n_q_heads * 4 : 0;
  Scratch sc{ctx, st};
  sc.cap = al(x_bytes) + 2 * al(o_bytes) + al(l_bytes) + q_project_scratch(ctx, M);
  CUDA_TRY(cudaMallocFromPoolAsync(&sc.base, sc.cap, ctx->mempool, st));
  char* base = static_cast<char*>(sc.base);
  void* x = base + sc.take(al(x_bytes));
  void* q = base + sc.take(al(o_bytes));
  void* out = base + sc.take(al(o_bytes));
  float* lse = lse_host ? reinterpret_cast<float*>(base + sc.take(al(l_bytes))) : nullptr;
  int launches = 0;
  cudaError_t ce = cudaMemcpyAsync(x, x_host, x_bytes, cudaMemcpyHostToDevice, st);
  if (ce == cudaSuccess && k_new_host != nullptr) {
    // the S new rows of each request, into rows S_kv - S .. of its S_kv
    const size_t row = (size_t)c.n_kv_heads * c.head_dim * 2;
    const size_t off = (size_t)(S_kv - S) * row;
    ce = cudaMemcpy2DAsync(static_cast<char*>(suffix_k) + off, (size_t)S_kv * row, k_new_host, (size_t)S * row,
                           (size_t)S * row, plan->n_req, cudaMemcpyHostToDevice, st);
    if (ce == cudaSuccess)
      ce = cudaMemcpy2DAsync(static_cast<char*>(suffix_v) + off, (size_t)S_kv * row, v_new_host, (size_t)S * row,
                             (size_t)S * row, plan->n_req, cudaMemcpyHostToDevice, st);
  }
  if (ce != cudaSuccess) e = fail(ATTUNER_ERR_CUDA, std::string("host-to-device copy: ") + cudaGetErrorString(ce));
  if (e == ATTUNER_OK)
    e = q_project_impl(ctx, plan, x, w_q, lora_a, lora_b, r, s, q_norm_w, S, S_kv, q, st, sc, launches);
  if (e == ATTUNER_OK)
    e = attend_launch(ctx, plan, q, suffix_k, suffix_v, S, S_kv, out, lse, st, nullptr, launches);
  if (e == ATTUNER_OK) {
    ce = cudaMemcpyAsync(out_host, out, o_bytes, cudaMemcpyDeviceToHost, st);
    if (ce == cudaSuccess && lse_host != nullptr)
      ce = cudaMemcpyAsync(lse_host, lse, l_bytes, cudaMemcpyDeviceToHost, st);
    if (ce != cudaSuccess) e = fail(ATTUNER_ERR_CUDA, std::string("device-to-host copy: ") + cudaGetErrorString(ce));
  }
  cudaFreeAsync(sc.base, st);
  ctx->last_launches = launches;
  return finish_call(ctx, e, st);
}

// ---------------------------------------------------------------------------
// APE-style read (App. C.2, APE paragraph): context and online attention
// computed separately, combined through calibrated log-sum-exp terms
// ---------------------------------------------------------------------------
extern "C" attuner_status attuner_attend_ape(attuner_ctx* ctx, const attuner_plan* plan, const void* q,
                                             const void* suffix_k, const void* suffix_v, int32_t S, int32_t S_kv,
                                             float temperature, float scale, void* out, float* lse_out,
                                             void* stream) {
  attuner_status e = check_common(ctx, plan, S, S_kv);
  if (e != ATTUNER_OK) return e;
  if (plan->max_o_rows > 0)
    return fail(ATTUNER_ERR_UNSUPPORTED, "attuner_attend_ape: plans with online spans between artifacts");
  CHECK_ARG(temperature > 0.f && scale > 0.f && std::isfinite(temperature) && std::isfinite(scale),
            "temperature and scale must be positive and finite");
  CHECK_ARG(out != nullptr && aligned16(out), "out must not be NULL and must be 16-byte aligned");
  if ((e = set_device(ctx)) != ATTUNER_OK) return e;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const attuner_config& c = ctx->cfg;
  const size_t rows = (size_t)plan->n_req * S * c.n_q_heads;
  auto al = [](size_t b) { return (b + 255) & ~size_t(255); };
  const size_t o_bytes = al(rows * c.head_dim * 2), l_bytes = al(rows * 4);
  void* base = nullptr;
  CUDA_TRY(cudaMallocFromPoolAsync(&base, 2 * (o_bytes + l_bytes), ctx->mempool, st));
  char* b = static_cast<char*>(base);
  void* o_ctx = b;
  float* lse_ctx = reinterpret_cast<float*>(b + o_bytes);
  void* o_on = b + o_bytes + l_bytes;
  float* lse_on = reinterpret_cast<float*>(b + 2 * o_bytes + l_bytes);
  int launches = 0;
  AttendVariant ctx_part;
  ctx_part.kv_part = 1;
  ctx_part.temperature = temperature;
  AttendVariant online_part;
  online_part.kv_part = 2;
  e = attend_launch(ctx, plan, q, suffix_k, suffix_v, S, S_kv, o_ctx, lse_ctx, st, nullptr, launches, ctx_part);
  if (e == ATTUNER_OK)
    e = attend_launch(ctx, plan, q, suffix_k, suffix_v, S, S_kv, o_on, lse_on, st, nullptr, launches, online_part);
  if (e == ATTUNER_OK) {
    ApeParams ap{};
    ap.o_ctx = static_cast<const __nv_bfloat16*>(o_ctx);
    ap.lse_ctx = lse_ctx;
    ap.o_on = static_cast<const __nv_bfloat16*>(o_on);
    ap.lse_on = lse_on;
    ap.out = static_cast<__nv_bfloat16*>(out);
    ap.lse_out = lse_out;
    ap.t_art = plan_dev(plan).t_art;
    ap.n_req = plan->n_req;
    ap.S = S;
    ap.Hq = c.n_q_heads;
    ap.D = c.head_dim;
    ap.scale = scale;
    const cudaError_t ce = launch_ape_combine(ap, st);
    if (ce != cudaSuccess) e = fail(ATTUNER_ERR_CUDA, std::string("APE combine launch failed: ") + cudaGetErrorString(ce));
    else ++launches;
  }
  cudaFreeAsync(base, st);
  ctx->last_launches = launches;
  return finish_call(ctx, e, st);
}

// ---------------------------------------------------------------------------
// misc
// ---------------------------------------------------------------------------
extern "C" attuner_status attuner_pool_info(const attuner_ctx* ctx, void** k_pool, void** v_pool,
                                            int32_t* used_blocks, int32_t* capacity_blocks) {
  CHECK_ARG(ctx != nullptr, "ctx must not be NULL");
  if (k_pool) *k_pool = ctx->kpool;
  if (v_pool) *v_pool = ctx->vpool;
  if (used_blocks) *used_blocks = ctx->used_blocks;
  if (capacity_blocks) *capacity_blocks = ctx->cfg.pool_blocks;
  return ATTUNER_OK;
}

extern "C" attuner_status attuner_sync_status(attuner_ctx* ctx, void* stream) {
  CHECK_ARG(ctx != nullptr, "ctx must not be NULL");
  attuner_status e = set_device(ctx);
  if (e != ATTUNER_OK) return e;
  CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  int h = 0;
  CUDA_TRY(cudaMemcpy(&h, ctx->d_status, sizeof(int), cudaMemcpyDeviceToHost));
  CUDA_TRY(cudaMemset(ctx->d_status, 0, sizeof(int)));
  if (h == ATTUNER_ERR_TIMEOUT) return fail(ATTUNER_ERR_TIMEOUT, "a kernel's bounded wait ran out");
  if (h == ATTUNER_ERR_DEVICE_CHECK) return fail(ATTUNER_ERR_DEVICE_CHECK, "a kernel rejected an out-of-range index");
  if (h != 0) return fail(ATTUNER_ERR_CUDA, "device status " + std::to_string(h));
  return ATTUNER_OK;
}

attuner_status att::finish_call(attuner_ctx* ctx, attuner_status e, cudaStream_t st) {
  if (e != ATTUNER_OK || !ctx->opt_sync_check) return e;
  return attuner_sync_status(ctx, st);
}

extern "C" attuner_status attuner_set_option(attuner_ctx* ctx, int32_t option, int64_t value) {
  CHECK_ARG(ctx != nullptr, "ctx must not be NULL");
  switch (option) {
    case ATTUNER_OPT_PREFILL_KERNEL:
      CHECK_ARG(value >= 0 && value <= 2, "prefill kernel must be 0, 1 or 2");
      ctx->opt_prefill = (int)value;
      return ATTUNER_OK;
    case ATTUNER_OPT_SPLIT_BLOCKS:
      CHECK_ARG(value >= 0 && value <= kMaxChunkBlocks, "split blocks must be in [0, 4096]");
      ctx->opt_split = (int)value;
      return ATTUNER_OK;
    case ATTUNER_OPT_WAIT_LIMIT:
      CHECK_ARG(value >= 0, "wait limit must be >= 0");
      ctx->wait_limit = value ? value : (1ll << 32);
      return ATTUNER_OK;
    case ATTUNER_OPT_QPROJ_SPLIT_K:
      CHECK_ARG(value == 0 || value == 1 || value == 2 || value == 4 || value == 8,
                "Q-projection split-K must be 0, 1, 2, 4 or 8");
      ctx->opt_qproj_split = (int)value;
      return ATTUNER_OK;
    case ATTUNER_OPT_QPROJ_ROWS:
      CHECK_ARG(value == 0 || value == 128 || value == 256, "Q-projection rows per CTA must be 0, 128 or 256");
      ctx->opt_qproj_rows = (int)value;
      return ATTUNER_OK;
    case ATTUNER_OPT_SPLIT_MERGE:
      CHECK_ARG(value >= 0 && value <= 2, "split merge must be 0, 1 or 2");
      ctx->opt_merge = (int)value;
      return ATTUNER_OK;
    case ATTUNER_OPT_SHARE_READS:
      CHECK_ARG(value >= 0 && value <= 2, "shared reads must be 0, 1 or 2");
      ctx->opt_share = (int)value;
      return ATTUNER_OK;
    case ATTUNER_OPT_SYNC_CHECK:
      ctx->opt_sync_check = value ? 1 : 0;
      return ATTUNER_OK;
    case ATTUNER_OPT_TEST_STUCK_WAIT:
      ctx->inject_stuck = value ? 1 : 0;
      return ATTUNER_OK;
    default:
      return fail(ATTUNER_ERR_INVALID_ARG, "unknown option " + std::to_string(option));
  }
}

extern "C" int32_t attuner_last_launch_count(const attuner_ctx* ctx) { return ctx ? ctx->last_launches : 0; }

extern "C" const char* attuner_last_error(void) { return g_err.c_str(); }
