/*
 * attuner.h - C ABI of the artifact-KV read path (libattuner.so).
 *
 * The library implements, for one decoder layer on one GB300 (sm_103a), the
 * request-time read of a frozen, independently cached artifact KV store as
 * the paper describes it:
 *
 *   Sec. 2, Eq. (1) and Eq. (full-vs-pic): every artifact A_j is encoded on
 *     its own, at local positions 0..L_j-1, and its K/V are stored for reuse;
 *     at request time the cached blocks are assembled in prompt order without
 *     re-encoding (App. A.3 "Cache construction and reuse", App. C.1 PIC).
 *   Sec. 3, Eq. (query-adaptation): the online tokens use the adapted query
 *     q = W^Q h + (alpha/r) B A h, then the model's original query RMSNorm
 *     and RoPE; artifact K/V never change.
 *   Sec. 2.2, Eq. (routing-oracle) and App. A.5 (Deployment): attention is
 *     softmax(q K^T / sqrt(d_k) + M_t) V with a causal mask and position ids
 *     of the assembled context.
 *
 * Conventions shared by every entry point
 *   - All tensors are row-major (last index fastest).  "bf16" is IEEE
 *     bfloat16 stored as 16-bit words.  Pointers are DEVICE pointers on the
 *     context's device unless the argument name ends in _host.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Device work is enqueued on it; the call returns before that
 *     work finishes unless the documentation says otherwise.
 *   - Every function returns an attuner_status and never throws.  On error a
 *     thread-local message is available from attuner_last_error().
 *   - The caller owns every input and output buffer; the library owns the
 *     context, the paged pool, plans and its per-call scratch (drawn from a
 *     stream-ordered memory pool of the context).
 *   - A context is not thread-safe: calls on one context must come from one
 *     host thread at a time.  Calls on different streams may overlap on the
 *     GPU; each call's scratch is private to it.
 *   - Device-side checks (bounded waits on mbarriers, block ids inside the
 *     pool) never trap: they set a status word in the context, which
 *     attuner_sync_status() returns and clears.
 */
#ifndef ATTUNER_H_
#define ATTUNER_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t attuner_status;

#define ATTUNER_OK                    0
#define ATTUNER_ERR_INVALID_ARG      (-1) /* a size, pointer or id is out of range      */
#define ATTUNER_ERR_OOM              (-2) /* pool full or a device allocation failed     */
#define ATTUNER_ERR_UNKNOWN_ARTIFACT (-3) /* an artifact id was never registered         */
#define ATTUNER_ERR_CUDA             (-4) /* a CUDA runtime or driver call failed        */
#define ATTUNER_ERR_TIMEOUT          (-5) /* a kernel's bounded wait ran out             */
#define ATTUNER_ERR_UNSUPPORTED      (-6) /* geometry the library has no kernel for     */
#define ATTUNER_ERR_DEVICE_CHECK     (-7) /* a kernel's bounds check rejected an index   */

/* Tokens per paged KV block.  Paging is this library's storage; the paper
 * only says that cached blocks are assembled (Sec. 2). */
#define ATTUNER_BLOCK_TOKENS 64

typedef struct attuner_config {
    int32_t hidden;        /* d_model of the projection input h (multiple of 64)          */
    int32_t n_q_heads;     /* Hq                                                           */
    int32_t n_kv_heads;    /* Hkv; Hq % Hkv == 0, G = Hq / Hkv in {1, 2, 4, 8}             */
    int32_t head_dim;      /* d in {64, 128}                                               */
    int32_t block_tokens;  /* must be ATTUNER_BLOCK_TOKENS                                 */
    int32_t pool_blocks;   /* capacity of the paged K/V pool, in blocks                    */
    float   rope_theta;    /* RoPE base (1e6 for Qwen3)                                    */
    float   rms_eps;       /* q RMSNorm epsilon (1e-6 for Qwen3)                           */
    int32_t device;        /* CUDA device ordinal the context lives on                     */
} attuner_config;

typedef struct attuner_ctx attuner_ctx;
typedef struct attuner_plan attuner_plan;

/* Create a context: allocates the paged K/V pool of cfg->pool_blocks blocks,
 * each [Hkv][64][d] bf16 for K and the same for V (16 KiB per block and head
 * at d = 128).  Errors: INVALID_ARG for an unsupported field, OOM, CUDA. */
attuner_status attuner_create(const attuner_config* cfg, attuner_ctx** out);

/* Free the context, its pool and every stream-ordered scratch it cached.
 * The caller must have finished all work it enqueued with this context.
 * Plans of the context not yet freed must not be used afterwards; freeing
 * them later is allowed (each releases its own device buffer then). NULL is
 * accepted.  Errors: none (always OK). */
attuner_status attuner_destroy(attuner_ctx* ctx);

/* Register one artifact (Sec. 2, Eq. full-vs-pic: Z^PIC = C(A | P_cache),
 * encoded alone at local positions 0..L-1, K already rotated there).
 *   k, v : [L, Hkv, d] bf16, device.  Copied into ceil(L/64) consecutive pool
 *          blocks on `stream`; the caller's buffers are free once that copy
 *          has run.
 *   Blocks are handed out in registration order by a bump allocator:
 *   artifact j owns blocks first_j .. first_j + ceil(L_j/64) - 1 with
 *   first_j = sum_{i<j} ceil(L_i/64), and artifact ids are 0, 1, 2, ...
 * Errors: INVALID_ARG (L outside [1, 2^30), NULL pointers), OOM (pool full). */
attuner_status attuner_register_artifact(attuner_ctx* ctx, const void* k, const void* v,
                                         int32_t L, void* stream, int32_t* artifact_id_out);

/* Assemble a batch of requests (Sec. 2 PIC box: cached blocks in prompt
 * order; App. A.3).  artifact_ids_host lists every request's artifacts in
 * runtime order, CSR-indexed by req_offsets_host[0..n_req] (host arrays).
 * Duplicates are allowed (assembled twice); an empty list is allowed (the
 * request then attends to its suffix only).  The plan holds, per request,
 * the block table (pool block, valid length) and the assembled index map
 * index_map[t] = block * 64 + slot for t in [0, T_art).  Synchronous: the
 * plan is on the device when the call returns.  A plan serves only the
 * context that assembled it, and only until that context's next
 * attuner_pool_reset: calls given another plan fail with INVALID_ARG.
 * Errors: INVALID_ARG, UNKNOWN_ARTIFACT, OOM, CUDA. */
attuner_status attuner_assemble(attuner_ctx* ctx, const int32_t* artifact_ids_host,
                                const int32_t* req_offsets_host, int32_t n_req,
                                attuner_plan** out);

/* A plan for a prompt layout whose online text interleaves with the cached
 * artifacts (App. "Prompt Construction and Artifact Boundaries": instructions,
 * separators and the question are processed online, only artifact spans are
 * cached).  items[] per request in prompt order: item >= 0 is an artifact id,
 * item < 0 an online span of -item tokens.  The request's online tokens live
 * in one online buffer in prompt order (x rows and suffix K/V rows): the spans'
 * rows first, then the final span (online rows sum(spans) .. S_kv - 1, the
 * suffix), so S_kv must be at least the spans' total.  The queries are the
 * last S online rows (S = S_kv for a whole prefill layer); each sits at its
 * index in the assembled sequence (App. A.5 position ids) and sees exactly the
 * assembled tokens up to it, and suffix K/V rows must be rotated at those same
 * positions (attuner_kv_project does so).  With no negative item this is
 * attuner_assemble.  Errors: as attuner_assemble, plus INVALID_ARG for more
 * than 2^22 online rows in the spans of one request. */
attuner_status attuner_assemble_layout(attuner_ctx* ctx, const int32_t* items_host,
                                       const int32_t* req_offsets_host, int32_t n_req,
                                       attuner_plan** out);

/* Copy a plan's layout to host arrays (for bit-exact tests).
 * sizes_inout[0..4] on input: capacities of block_table, valid_len,
 * index_map, token_art, token_off (elements); on output: the lengths used,
 * and sizes_inout[5] = number of requests.  Per request the arrays are
 * concatenated in request order (blocks first by request, then tokens).
 * Any output pointer may be NULL to skip it.  Errors: INVALID_ARG when a
 * capacity is too small. */
attuner_status attuner_plan_export(const attuner_plan* plan, int32_t* block_table_host,
                                   int32_t* valid_len_host, int32_t* index_map_host,
                                   int32_t* token_art_host, int32_t* token_off_host,
                                   int64_t* sizes_inout);

/* Per-request assembled artifact length T_art (host array of n_req), the
 * offset of the suffix positions (App. A.5).  Errors: INVALID_ARG for NULL
 * pointers or an n_req other than the plan's. */
attuner_status attuner_plan_t_art(const attuner_plan* plan, int32_t* t_art_host, int32_t n_req);

/* Free a plan. The caller must have finished all work that reads it. Its
 * device buffer goes back to the context, which reuses a few such buffers
 * for later assemblies instead of allocating.  NULL is accepted.  Errors:
 * none (always OK). */
attuner_status attuner_plan_free(attuner_plan* plan);

/* Adapted query of the online tokens (Sec. 3, Eq. query-adaptation, then
 * the query RMSNorm and RoPE):
 *   q[m] = RoPE( RMSNorm_head( W_q x_m + s * B (A x_m) ) * q_norm_w, pos_m )
 *   x        [n_req, S, hidden] bf16
 *   w_q      [Hq*d, hidden] bf16 (output x input, as stored by HF q_proj)
 *   lora_a   [r, hidden] bf16, lora_b [Hq*d, r] bf16; r in {0, 8, 16, ..., 64};
 *            r = 0 or NULL A/B is the merged deployment form (App. A.5).
 *            A x is rounded to bf16 before B is applied (as a bf16 PEFT layer
 *            does); everything else accumulates in fp32.
 *   q_norm_w [d] bf16; eps and theta come from the context config.
 *   pos_m    = T_art(req) + (S_kv - S) + i for suffix token i.
 *   q_out    [n_req, S, Hq, d] bf16.
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
attuner_status attuner_q_project(attuner_ctx* ctx, const attuner_plan* plan, const void* x,
                                 const void* w_q, const void* lora_a, const void* lora_b,
                                 int32_t r, float s, const void* q_norm_w, int32_t S,
                                 int32_t S_kv, void* q_out, void* stream);

/* Attention of the online queries over the assembled artifact KV followed
 * by the suffix's own KV (Eq. routing-oracle with the causal mask M_t):
 *   q        [n_req, S, Hq, d] bf16 (already normalised and rotated)
 *   suffix_k, suffix_v [n_req, S_kv, Hkv, d] bf16, K rotated at positions
 *            T_art .. T_art + S_kv - 1.
 *   Query i of a request sees all T_art artifact tokens and suffix keys
 *   j <= (S_kv - S) + i; q head h reads KV head h / (Hq/Hkv).
 *   out      [n_req, S, Hq, d] bf16, softmax(q k^T / sqrt(d)) v.
 *   lse_out  [n_req, S, Hq] fp32 natural-log softmax denominator, or NULL.
 * A plan with no artifacts gives plain causal attention over the suffix.
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
attuner_status attuner_attend(attuner_ctx* ctx, const attuner_plan* plan, const void* q,
                              const void* suffix_k, const void* suffix_v, int32_t S,
                              int32_t S_kv, void* out, float* lse_out, void* stream);

/* attuner_attend for callers that cannot allocate GPU memory (no
 * counterpart in the paper).  Some callers own the whole device: a serving
 * engine whose allocator reserves the GPU up front, or a runtime that bars
 * other libraries from cudaMalloc or stream-ordered pools because such an
 * allocation can synchronise the device or fail in the middle of a request.
 * This call runs the same kernels with the same split-KV decomposition as
 * attuner_attend, with the same arguments and results, but keeps the split
 * partial results in one fixed 32 MiB array in device memory that the library
 * declares at file scope; it calls no allocator of any kind.
 *   - The array exists on every GPU that loads the library until the process
 *     exits, one copy per CUDA context.  The first call in each context (so
 *     once per device, and again after cudaDeviceReset) looks up its device
 *     address (cudaGetSymbolAddress), which may load the library's module:
 *     make that first call outside any stream capture.
 *   - Every call in a context shares the array and it keeps the last call's
 *     contents (nothing in it needs to start at zero; the call clears the
 *     arrival counters it keeps there with cudaMemsetAsync on `stream`).
 *     Calls whose kernels overlap on the GPU race on it: order them (one
 *     stream, or events).
 *   - A call whose partial results would need more than 32 MiB
 *     (n_split_ctas * rows_per_cta * (d + 1) * 4 bytes, plus 4 bytes per
 *     (request, KV head, row tile) for the tcgen05 kernel) is rejected with
 *     INVALID_ARG before anything is launched; use attuner_attend for it.
 * Errors: as attuner_attend, plus INVALID_ARG for a call beyond the limit. */
attuner_status attuner_attend_static_scratch(attuner_ctx* ctx, const attuner_plan* plan,
                                             const void* q, const void* suffix_k,
                                             const void* suffix_v, int32_t S, int32_t S_kv,
                                             void* out, float* lse_out, void* stream);

/* The suffix tokens' own keys and values (the layer's remaining online
 * computation).  The adaptation changes W^Q only (Sec. 3), so K and V come
 * from the base model's projections: for request r and new suffix token i < S
 * (query position T_art(r) + S_kv - S + i, App. A.5)
 *   suffix_k[r, S_kv - S + i, h, :] = RoPE(RMSNorm(x[r, i] W_k,h^T) * k_norm_w, pos)
 *   suffix_v[r, S_kv - S + i, h, :] = x[r, i] W_v,h^T
 *   x        [n_req, S, hidden] bf16
 *   w_k, w_v [Hkv*d, hidden] bf16 (output x input)
 *   k_norm_w [d] bf16
 *   suffix_k, suffix_v [n_req, S_kv, Hkv, d] bf16: only the last S token rows
 *            of each request are written, so a decode step (S = 1) appends
 *            one token to KV the caller keeps.
 * Errors: INVALID_ARG, CUDA. */
attuner_status attuner_kv_project(attuner_ctx* ctx, const attuner_plan* plan, const void* x,
                                  const void* w_k, const void* w_v, const void* k_norm_w, int32_t S,
                                  int32_t S_kv, void* suffix_k, void* suffix_v, void* stream);

/* The whole path (Sec. 3, Eq. query-adaptation, then Sec. 2.2, Eq.
 * routing-oracle): attuner_q_project into stream-ordered scratch, then
 * attuner_attend.  Arguments as in those two calls.  Errors: as those two
 * calls, plus CUDA when the scratch cannot be drawn from the context's pool. */
attuner_status attuner_query_attend(attuner_ctx* ctx, const attuner_plan* plan, const void* x,
                                    const void* w_q, const void* lora_a, const void* lora_b,
                                    int32_t r, float s, const void* q_norm_w,
                                    const void* suffix_k, const void* suffix_v, int32_t S,
                                    int32_t S_kv, void* out, float* lse_out, void* stream);

/* The whole path for a step whose new inputs and whose output live in HOST
 * memory (the request-time path of Sec. 3 Eq. query-adaptation and Sec. 2.2
 * Eq. routing-oracle, as attuner_query_attend).  On `stream`, in order: the
 * new tokens' hidden states are copied from host memory into stream-ordered
 * device scratch; when k_new_host and v_new_host are given, the new tokens'
 * own K/V rows are copied into rows S_kv - S .. S_kv - 1 of each request of
 * suffix_k / suffix_v; the projection and the attention run; O (and the LSE
 * when lse_host is given) are copied back to host memory.
 *   x_host      [n_req, S, hidden] bf16, host memory
 *   k_new_host, v_new_host  [n_req, S, Hkv, d] bf16, host memory, RoPE'd at
 *               the tokens' positions; both NULL when the caller's device
 *               suffix K/V already hold them (e.g. from attuner_kv_project)
 *   suffix_k, suffix_v  [n_req, S_kv, Hkv, d] bf16, device memory: the rows
 *               before the new tokens are the request's resident online KV
 *   out_host    [n_req, S, Hq, d] bf16, host memory; lse_host [n_req, S, Hq]
 *               fp32, host memory, or NULL
 *   w_q, lora_a, lora_b, q_norm_w: device memory, as in attuner_q_project
 * The call returns once everything is enqueued; out_host and lse_host hold
 * the result when the stream reaches the end of the call (an event recorded
 * after it, or a stream synchronisation).  The host buffers must stay valid
 * and unchanged until then.  Pinned (page-locked) host memory makes the
 * copies asynchronous; with pageable memory the driver stages them and the
 * call may block.  Errors: as attuner_query_attend, plus INVALID_ARG for a
 * NULL x_host, out_host, suffix_k or suffix_v, or only one of k_new_host and
 * v_new_host given. */
attuner_status attuner_query_attend_host(attuner_ctx* ctx, const attuner_plan* plan,
                                         const void* x_host, const void* w_q, const void* lora_a,
                                         const void* lora_b, int32_t r, float s, const void* q_norm_w,
                                         const void* k_new_host, const void* v_new_host,
                                         void* suffix_k, void* suffix_v, int32_t S, int32_t S_kv,
                                         void* out_host, float* lse_host, void* stream);

/* Keys stored before RoPE, rotated to their target positions at assembly:
 * the read of the paper's EPIC baseline (App. C.2 "Training-Free Baselines",
 * EPIC paragraph: cached keys kept un-rotated and rotated to their place in
 * the assembled prompt).  The plan's artifacts must have been registered
 * with keys BEFORE RoPE; artifact token t of a request is rotated at its
 * assembled position (the request's artifact tokens before it, in runtime
 * order from 0: the position a full prefill would give it).  One kernel on
 * `stream` writes the rotated keys into a buffer the plan owns
 * ([n_blocks][Hkv][64][d] bf16, freed by attuner_plan_free); from then on
 * every attention call with this plan reads its artifact keys there (values
 * still from the pool), and queries and suffix keys are as for the plain
 * read.  Calling it again re-rotates into the same buffer.  The call
 * allocates the buffer (cudaMalloc) on first use and returns once the
 * rotation has finished (it synchronises `stream`).
 * Errors: INVALID_ARG (NULL, foreign or stale plan), UNSUPPORTED (a plan with
 * online spans between artifacts), OOM, CUDA; DEVICE_CHECK through
 * attuner_sync_status when a block id is out of the pool. */
attuner_status attuner_plan_rotate_keys(attuner_ctx* ctx, attuner_plan* plan, void* stream);

/* The read of the paper's APE baseline (App. C.2, APE paragraph): attention
 * over the cached context and over the online tokens computed separately,
 * the context's logits divided by `temperature`, and the two results
 * combined through calibrated log-sum-exp terms.  The paper uses
 * temperature 0.9 and scale 0.9 without stating how the scale enters; here
 * it multiplies the context's log-sum-exp (its softmax denominator Z_c counts
 * as Z_c^scale):
 *   (o_c, lse_c) = softmax(q k_art^T / (temperature sqrt(d))) v_art, every
 *                  artifact token visible;
 *   (o_o, lse_o) = causal attention over the suffix keys j <= (S_kv - S) + i;
 *   out = (e^(scale lse_c) o_c + e^(lse_o) o_o) / (e^(scale lse_c) + e^(lse_o)),
 *   lse_out = log(e^(scale lse_c) + e^(lse_o)); a request without artifacts
 *   takes o_o and lse_o.
 * Arguments and layouts as in attuner_attend; temperature = scale = 1 gives
 * attuner_attend's result.  Three launches (context part, online part,
 * combine) with their two partial results in stream-ordered scratch.
 * Errors: INVALID_ARG (also temperature or scale not positive and finite),
 * UNSUPPORTED (a plan with online spans between artifacts), CUDA. */
attuner_status attuner_attend_ape(attuner_ctx* ctx, const attuner_plan* plan, const void* q,
                                  const void* suffix_k, const void* suffix_v, int32_t S, int32_t S_kv,
                                  float temperature, float scale, void* out, float* lse_out,
                                  void* stream);

/* Warm-cache load (the "CPU RAM cache lookup and GPU transfer" stage of the
 * paper's time-to-first-token, Sec. 5 / App. A.3: encoded artifacts kept in
 * host memory and moved to the GPU when a request needs them).  Registers n
 * artifacts whose K/V live in PINNED host memory (cudaMallocHost /
 * cudaHostAlloc / a pinned torch tensor) in one kernel that reads them over
 * the CPU-GPU link and writes their paged pool blocks, on `stream`; run it on
 * a second stream to overlap it with attuner_q_project, and make the attention
 * stream wait for it.
 *   k_host[i], v_host[i] : [L[i], Hkv, d] bf16, pinned host memory, 16-byte
 *                          aligned; the caller keeps them alive and unchanged
 *                          until the copy has run.
 *   ids_out[i]           : artifact ids, allocated as by
 *                          attuner_register_artifact, in order.
 *   1 <= n <= ATTUNER_MAX_HOST_BATCH.
 * Errors: INVALID_ARG (n out of range, L outside [1, 2^30), NULL or unaligned pointers,
 * memory that is not pinned host memory), OOM (pool full; nothing is
 * registered then). */
#define ATTUNER_MAX_HOST_BATCH 64
attuner_status attuner_register_artifacts_host(attuner_ctx* ctx, int32_t n, const void* const* k_host,
                                               const void* const* v_host, const int32_t* L,
                                               void* stream, int32_t* ids_out);

/* Forget every registered artifact: the pool is empty again and the next
 * artifact gets id 0 and block 0 (a serving loop's eviction of the whole warm
 * set).  Plans made before are rejected afterwards (INVALID_ARG), and the
 * caller must not reset while kernels that read the pool are still running.
 * Errors: INVALID_ARG for a NULL context. */
attuner_status attuner_pool_reset(attuner_ctx* ctx);

/* The paged pool: device base pointers of K and V ([pool_blocks][Hkv][64][d]
 * bf16 each), blocks in use and capacity.  Any output may be NULL.  The
 * pointers stay owned by the context.  Errors: INVALID_ARG for a NULL context. */
attuner_status attuner_pool_info(const attuner_ctx* ctx, void** k_pool, void** v_pool,
                                 int32_t* used_blocks, int32_t* capacity_blocks);

/* Synchronise `stream`, then return and clear the device status word.
 * Errors: TIMEOUT (a bounded wait ran out), DEVICE_CHECK (an index failed a
 * bounds check), CUDA if the synchronisation itself failed, INVALID_ARG for a
 * NULL context. */
attuner_status attuner_sync_status(attuner_ctx* ctx, void* stream);

/* Tuning and test options (value 0 restores the default):
 *   ATTUNER_OPT_PREFILL_KERNEL  0 auto, 1 tcgen05 tile kernel, 2 warp-MMA kernel
 *   ATTUNER_OPT_SPLIT_BLOCKS    KV blocks per split-KV chunk (0 = automatic)
 *   ATTUNER_OPT_WAIT_LIMIT      clock cycles a device wait may spin before it
 *                               gives up and sets TIMEOUT (0 = about 2 s)
 *   ATTUNER_OPT_QPROJ_SPLIT_K   CTAs (a thread-block cluster: 1, 2, 4 or 8) that
 *                               split the K dimension of one projection tile
 *                               (0 = chosen by the library's cost model)
 *   ATTUNER_OPT_QPROJ_ROWS      query rows per projection CTA: 128 or 256
 *                               (0 = chosen by the cost model).  A pair of these
 *                               two options that no kernel shape supports for
 *                               the context's head size and the call's LoRA
 *                               rank makes the projection calls fail with
 *                               INVALID_ARG
 *   ATTUNER_OPT_SPLIT_MERGE     how the tcgen05 kernel merges the split-KV
 *                               chunks of a row tile: 0 auto (cost model),
 *                               1 independent CTAs merged through global memory
 *                               by the last one to finish, 2 one thread-block
 *                               cluster per row tile (2 or 4 chunks) merged
 *                               through distributed shared memory (global
 *                               memory where such clusters cannot be
 *                               co-resident on the device)
 *   ATTUNER_OPT_SHARE_READS     shared artifact reads of the decode kernel
 *                               (the warp-MMA kernel, at most 16 packed query
 *                               rows per request): one CTA reads a chunk of an
 *                               artifact for every request of a group of
 *                               requests that use it, each request's partial
 *                               results merged afterwards.  0 auto (where it
 *                               saves 10 % or more of the block reads), 1 off,
 *                               2 wherever it applies: every query sees every
 *                               artifact (no online spans, or every query row
 *                               in its request's final online span, as a
 *                               decode token is), keys not rotated at assembly,
 *                               at least two requests' rows per CTA, at most
 *                               511 distinct artifacts in the plan
 *   ATTUNER_OPT_SYNC_CHECK      0 off, 1 every compute call reports the device
 *                               status itself (see below)
 *   ATTUNER_OPT_TEST_STUCK_WAIT see below */
#define ATTUNER_OPT_PREFILL_KERNEL 1
#define ATTUNER_OPT_SPLIT_BLOCKS   2
#define ATTUNER_OPT_WAIT_LIMIT     3
#define ATTUNER_OPT_QPROJ_SPLIT_K  4
#define ATTUNER_OPT_SPLIT_MERGE    5
#define ATTUNER_OPT_QPROJ_ROWS     7
#define ATTUNER_OPT_SHARE_READS    8
/* Debug check: while non-zero, attuner_q_project, attuner_kv_project,
 * attuner_attend, attuner_attend_static_scratch and attuner_query_attend
 * synchronise their stream before returning and return the device status as
 * their own (TIMEOUT, DEVICE_CHECK; the status word is cleared), as
 * attuner_sync_status would.  Not for calls captured into a CUDA graph. */
#define ATTUNER_OPT_SYNC_CHECK     6
/* Test hook (failure detection without a GPU fault): while non-zero, one
 * role of every attention launch waits on an mbarrier that nothing arrives
 * at; its bounded wait runs out, the kernel drains its own copies, frees its
 * tensor memory and returns, and attuner_sync_status() reports TIMEOUT. */
#define ATTUNER_OPT_TEST_STUCK_WAIT 1000
/* Set one option of the context; it applies to the calls that follow.
 * Errors: INVALID_ARG for a NULL context, an unknown option or a value out of
 * its range. */
attuner_status attuner_set_option(attuner_ctx* ctx, int32_t option, int64_t value);

/* Number of kernel launches the last call on this context enqueued (0 for a
 * NULL context). */
int32_t attuner_last_launch_count(const attuner_ctx* ctx);

/* Message of the last error on this host thread ("" if none). */
const char* attuner_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* ATTUNER_H_ */
