// attn_tc.cu - K2: attention of the online queries over the assembled
// artifact KV followed by the suffix KV (Sec. 2.2 Eq. routing-oracle with
// the causal mask M_t; App. A.5: SDPA with position ids of the assembled
// context), as a tcgen05 / TMEM / TMA flash-attention kernel.
//
// One CTA = 256 "packed" query rows of one request and one KV head, as two
// 128-row query tiles Q0 and Q1 (packed row = token * G + head_in_group: the
// G query heads that share a KV head are stacked into the MMA M dimension),
// and one split-KV chunk of the request's virtual block list (artifact blocks
// from the block table in runtime order, then 64-token chunks of the suffix).
//
// Per 128-key tile j (two 64-token blocks, each one TMA box per 64 columns):
//   S_i = Q_i K_j^T     tcgen05.mma M=128 N=128 K=D, A and B from SMEM -> TMEM
//   P_i = exp2(S_i * log2(e)/sqrt(D) - m_i)    softmax warpgroup i, written as
//                       bf16 back into the TMEM columns of S_i
//   O_i += P_i V_j      tcgen05.mma M=128 N=D K=128, A = P_i from TMEM, B = V
// The single MMA thread issues  PV_0(j), QK_0(j+1), PV_1(j), QK_1(j+1), so
// each softmax warpgroup works on its tile while the tensor pipe runs the
// other tile's products: every K/V tile feeds 4 MMAs, and the softmax of a
// tile has the time of two MMAs to finish.  A commit after QK_i(j+1) also
// covers every earlier MMA, so one barrier per tile tells softmax i that S_i
// is ready, that PV_i(j) has consumed P_i and that O_i is current.  The
// running max only moves when it grows by more than 2^8 (then O_i in TMEM is
// rescaled), so most tiles need no O round trip.
//
// Warpgroup 0 (warps 0..3): softmax of Q0; warpgroup 1 (warps 4..7): softmax
// of Q1 (one query row per thread = one TMEM lane; warp w reaches lanes
// 32*(w%4)..+31).  Warpgroup 2: warp 8 TMA producer, warp 9 TMEM owner and
// single-thread MMA issuer, warps 10..11 idle.  The block is launched with
// 384 threads x 168 registers = 64512; warpgroup 2 drops to kCtrlRegs and the
// softmax warpgroups rise to kSoftRegs: 128 x kCtrlRegs + 256 x kSoftRegs
// <= 64512, so every score of a tile stays in registers.
#include <math.h>

#include <cuda_fp16.h>

#include "kernels.h"

namespace att {

template <int D>
struct TcLayout {
  static constexpr int NH = D / 64;                 // 64-column (128-byte) halves
  static constexpr int NS = 2;                      // K and V pipeline stages
  static constexpr int HALF = 128 * 128;            // 128 rows x 128 B
  static constexpr int Q_OFF = 0;                   // Q0 then Q1, NH halves each
  static constexpr int K_OFF = Q_OFF + 2 * NH * HALF;
  static constexpr int V_OFF = K_OFF + NS * NH * HALF;
  static constexpr int BAR_OFF = V_OFF + NS * NH * HALF;
  static constexpr int LIST_OFF = BAR_OFF + 1024;
  static constexpr int XLSE_OFF = LIST_OFF + kMaxChunkBlocks * 4;   // cluster merge: LSE out + 3 in
  static constexpr int SMEM_MIN = XLSE_OFF + 4 * kTcRows * 4 + 1024;
  // at least 116 KiB so that two CTAs never share an SM (each holds all of TMEM)
  static constexpr int SMEM = SMEM_MIN > 118784 ? SMEM_MIN : 118784;
  static constexpr uint32_t TMEM_COLS = 512;        // S0/P0 | S1/P1 | O0 | O1
};

__device__ __forceinline__ uint32_t s_col_of(int qt) { return qt ? 128u : 0u; }
__device__ __forceinline__ uint32_t o_col_of(int qt) { return qt ? 384u : 256u; }

constexpr int kProducerWarp = 8, kMmaWarp = 9;
constexpr int kCtrlRegs = 96, kSoftRegs = 200;
static_assert(128 * kCtrlRegs + 256 * kSoftRegs <= 384 * 168, "register split exceeds the launch budget");

enum : int {
  B_Q = 0, B_KF = 1, B_VF = 3, B_KE = 5, B_VE = 7, B_SF = 9, B_PF = 11,
  B_O = 13, B_DRAIN = 14, B_NEVER = 15,
  B_MF = 16, B_ME = 24,   // split merge: full / empty barriers of up to 8 staging buffers
  B_COUNT = 32
};

// D[tmem] (+)= A[tmem] * B[smem desc]: A (M x 16 bf16 per step) read from TMEM,
// lane = row, each 32-bit column two consecutive K elements.
ATT_DEV void umma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// load the K (or V) half-tiles of block slot `e` into `dst` (64-column halves
// at +HALF); an artifact slot reads rows kslot_row.. of `kslot` instead of its
// pool block when `kslot` is given (keys rotated at assembly)
template <int D>
__device__ __forceinline__ void load_slot(uint32_t dst, int e, const CUtensorMap* pool,
                                          const CUtensorMap* suf, uint32_t bar, int kvh, int Hkv,
                                          int req, int pool_rows, const CUtensorMap* kslot = nullptr,
                                          int kslot_row = 0) {
  using L = TcLayout<D>;
#pragma unroll
  for (int h = 0; h < L::NH; ++h) {
    if (e < 0) {
      tma_load_4d(dst + h * L::HALF, suf, bar, h * 64, kvh, slot_row0(e), req);
    } else if ((e & 127) != 0) {
      if (kslot != nullptr) {
        tma_load_2d(dst + h * L::HALF, kslot, bar, h * 64, kslot_row);
      } else {
        const int blk = e >> 7;
        tma_load_2d(dst + h * L::HALF, pool, bar, h * 64, (blk * Hkv + kvh) * kBlockTokens);
      }
    } else {
      // no block: a box entirely past the end of the pool reads zeros
      tma_load_2d(dst + h * L::HALF, pool, bar, h * 64, pool_rows);
    }
  }
}

// -inf for keys past n_vis in a 64-key slot
__device__ __forceinline__ void mask_tail(float* v, int n_vis) {
#pragma unroll
  for (int c = 0; c < 64; ++c) v[c] = (c < n_vis) ? v[c] : -INFINITY;
}

// Which (request, KV head, row tile, split) a CTA owns, and its KV chunk size
// in blocks.  Independent splits: CTAs in [request][split][kv head][row tile]
// order.  Cluster mode: one cluster per (request, kv head, row tile), split =
// rank, every request cut into `cluster` chunks of whole 128-key tiles.
struct TcCta {
  int req, rt, kvh, split, nsplit, chunk;
};
__device__ __forceinline__ TcCta tc_cta(const AttnParams& p, int cta) {
  TcCta c;
  if (p.work.cluster > 0) {
    const int ns = p.work.cluster, unit = cta / ns, per_req = p.Hkv * p.work.row_tiles;
    c.split = cta % ns;
    c.nsplit = ns;
    c.req = unit / per_req;
    const int rem = unit % per_req;
    c.rt = rem % p.work.row_tiles;
    c.kvh = rem / p.work.row_tiles;
    int lo, hi;
    kv_part_range(p.kv_part, p.plan.blk_off[c.req + 1] - p.plan.blk_off[c.req],
                  (p.S_kv + kBlockTokens - 1) / kBlockTokens, lo, hi);
    const int nv = hi - lo;
    c.chunk = (((nv + ns - 1) / ns) + 1) & ~1;
  } else {
    c.req = find_req(p.work, cta);
    int rel = cta - p.work.base[c.req];
    c.rt = rel % p.work.row_tiles;
    rel /= p.work.row_tiles;
    c.kvh = rel % p.Hkv;
    c.split = rel / p.Hkv;
    c.nsplit = p.work.nsplit[c.req];
    c.chunk = p.work.chunk_blocks;
  }
  return c;
}

// the CTA index, read so that the compiler recomputes what derives from it
// instead of keeping it in registers across the main loop
__device__ __forceinline__ int cta_index_fresh() {
  int v;
  asm volatile("mov.u32 %0, %%ctaid.x;" : "=r"(v));
  return v;
}

// bf16 store of N columns of one output row, from column c0 on, scaled
template <int D, int N>
__device__ __forceinline__ void store_cols(__nv_bfloat16* out, long long orow, int c0, const float* o, float scale) {
  uint4* dst = reinterpret_cast<uint4*>(out + orow * D + c0);
#pragma unroll
  for (int k = 0; k < N / 8; ++k)
    dst[k] = make_uint4(pack_bf16(o[8 * k] * scale, o[8 * k + 1] * scale),
                        pack_bf16(o[8 * k + 2] * scale, o[8 * k + 3] * scale),
                        pack_bf16(o[8 * k + 4] * scale, o[8 * k + 5] * scale),
                        pack_bf16(o[8 * k + 6] * scale, o[8 * k + 7] * scale));
}

// Cluster-mode merge of the NS split-KV chunks of a row tile (one CTA per
// chunk, cluster rank = split).  CTA `split` produces columns
// [split, split + 1) x D/NS of all 256 rows.  Each CTA stages the other CTAs'
// columns of its normalised O and its LSE, and pushes them into the peers'
// shared memory with bulk copies (the copy engine moves distributed shared
// memory about twice as fast as loads from a peer do); its own columns stay
// in tensor memory.  The pushed columns travel as fp16 pairs divided by a
// power of 2 per row (the one just above the row's largest magnitude, sent
// beside them), so no value overflows and each keeps 11 bits relative to its
// row's largest, finer than the bf16 rounding of the output; half the bytes
// of fp32 halve the transfer, the epilogue's largest part.  The chunks are
// summed in split order with the same arithmetic whichever CTA finishes
// first, and the merged [256][D/NS] bf16 tile leaves through one TMA tensor
// store (rows past the last token clipped by the map) instead of 64-byte
// pieces per row.  The loops over peers stay rolled: this code runs once per
// CTA, cold, and its instruction fetch costs more than its arithmetic.
template <int D, int NS>
__device__ __forceinline__ void tc_cluster_merge(const AttnParams& p, uint8_t* smem, const TcCta& ce,
                                                 uint32_t o_col, bool ok, int ntile, float inv_l, float lse,
                                                 long long orow, bool row_ok) {
  using L = TcLayout<D>;
  constexpr int CW = D / NS;                            // output columns per CTA
  // one chunk's columns of all rows as fp16 pairs [CW/2][256], then a power-of-2 scale per row
  constexpr uint32_t kVals = kTcRows * CW * 2;
  constexpr uint32_t kSlot = kVals + kTcRows * 4;
  static_assert(CW % 16 == 0 && 2 * (NS - 1) * kSlot <= (uint32_t)L::BAR_OFF, "staging and receive slots");
  static_assert(NS <= 4, "LSE slots");
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR_OFF);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 520);
  const uint32_t mbar = smem_u32(&bars[B_MF]);
  const int split = ce.split, erow = threadIdx.x;
  uint8_t* src = smem;                                  // NS-1 outgoing slots, peer order
  uint8_t* rcv = smem + (NS - 1) * kSlot;               // NS-1 incoming slots, split order
  float* src_lse = reinterpret_cast<float*>(smem + L::XLSE_OFF);
  float* rcv_lse = src_lse + kTcRows;
  auto own_cols = [&](int c0, float* v) {
    if (ok && ntile > 0) {
      if constexpr (CW >= 32) {
#pragma unroll
        for (int c = 0; c < CW; c += 32) tmem_ld32(o_col + c0 + c, v + c);
        tc_wait_ld();
      } else {
        float t[32];
        tmem_ld32(o_col + (c0 & ~31), t);
        tc_wait_ld();
        const bool hi = (c0 & 31) != 0;
#pragma unroll
        for (int k = 0; k < CW; ++k) v[k] = hi ? t[16 + k] : t[k];
      }
#pragma unroll
      for (int k = 0; k < CW; ++k) v[k] *= inv_l;
    } else {
#pragma unroll
      for (int k = 0; k < CW; ++k) v[k] = 0.f;
    }
  };
  if (threadIdx.x == 0) mbar_expect_tx(mbar, (NS - 1) * (kSlot + kTcRows * 4));
#pragma unroll 1
  for (int t = 0; t < NS; ++t) {
    if (t == split) continue;
    float v[CW];
    own_cols(t * CW, v);
    float amax = 0.f;
#pragma unroll
    for (int k = 0; k < CW; ++k) amax = fmaxf(amax, fabsf(v[k]));
    // scale = the power of 2 just above the row's largest magnitude: v / scale in [-1, 1]
    const int ex = (__float_as_int(amax) >> 23) & 0xff;
    const float scale = (amax > 0.f && ex < 254) ? __int_as_float((ex + 1) << 23) : 1.f;
    const float inv = 1.f / scale;
    uint8_t* slot = src + (t < split ? t : t - 1) * kSlot;
    uint32_t* dst = reinterpret_cast<uint32_t*>(slot) + erow;
#pragma unroll
    for (int c = 0; c < CW / 2; ++c) {
      const __half2 h = __floats2half2_rn(v[2 * c] * inv, v[2 * c + 1] * inv);
      dst[c * kTcRows] = *reinterpret_cast<const uint32_t*>(&h);
    }
    reinterpret_cast<float*>(slot + kVals)[erow] = scale;
  }
  src_lse[erow] = lse;
  fence_proxy_async_smem();
  cluster_sync_all();   // 1: every CTA of the cluster has staged; all main loops are over
  if (threadIdx.x == 0) {
#pragma unroll 1
    for (int t = 0; t < NS; ++t) {
      if (t == split) continue;
      const uint32_t at = (split < t ? split : split - 1);   // this CTA's slot at peer t
      const uint32_t cbar = dsmem_addr(mbar, t);
      bulk_push_dsmem(dsmem_addr(smem_u32(rcv) + at * kSlot, t), smem_u32(src) + (t < split ? t : t - 1) * kSlot,
                      kSlot, cbar);
      bulk_push_dsmem(dsmem_addr(smem_u32(rcv_lse) + at * kTcRows * 4, t), smem_u32(src_lse), kTcRows * 4, cbar);
    }
  }
  // this CTA's own columns while the peers' arrive
  float acc[CW];
  own_cols(split * CW, acc);
  // Every CTA waits for its incoming copies, also after an abort: the peers
  // issue them unconditionally, and none may land after this CTA has exited.
  // One answer for the whole CTA, so the barrier below is passed by all.
  const bool got = __all_sync(0xffffffffu, mbar_drain(mbar, 0, p.status));
  if (!got && (threadIdx.x & 31) == 0) *abort_flag = 1;
  asm volatile("bar.sync 1, 256;" ::: "memory");
  const bool merge = *abort_flag == 0;
  // output tile [256 rows][CW] bf16 after the slots, in the tensor map's swizzle
  constexpr uint32_t kOutOff = (2 * (NS - 1) * kSlot + 1023) & ~1023u;
  static_assert(kOutOff + kTcRows * CW * 2 <= (uint32_t)L::BAR_OFF, "output tile");
  if (merge) {
    auto lse_of = [&](int k) { return (k == split) ? lse : rcv_lse[(k < split ? k : k - 1) * kTcRows + erow]; };
    float mx = -INFINITY;
#pragma unroll 1
    for (int k = 0; k < NS; ++k) mx = fmaxf(mx, lse_of(k));
    // chunks in split order; the own chunk's term first computed into acc[] is
    // rebuilt in order: acc = sum_k w_k * chunk_k
    float own[CW];
#pragma unroll
    for (int c = 0; c < CW; ++c) { own[c] = acc[c]; acc[c] = 0.f; }
    float wsum = 0.f;
#pragma unroll 1
    for (int k = 0; k < NS; ++k) {
      const float lk = lse_of(k);
      const float w = (lk == -INFINITY) ? 0.f : __expf(lk - mx);
      wsum += w;
      if (k == split) {
#pragma unroll
        for (int c = 0; c < CW; ++c) acc[c] = __fmaf_rn(w, own[c], acc[c]);
      } else {
        const uint8_t* slot = rcv + (k < split ? k : k - 1) * kSlot;
        const uint32_t* r = reinterpret_cast<const uint32_t*>(slot) + erow;
        const float wk = w * reinterpret_cast<const float*>(slot + kVals)[erow];
#pragma unroll
        for (int c = 0; c < CW / 2; ++c) {
          const uint32_t bits = r[c * kTcRows];
          const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&bits));
          acc[2 * c] = __fmaf_rn(wk, f.x, acc[2 * c]);
          acc[2 * c + 1] = __fmaf_rn(wk, f.y, acc[2 * c + 1]);
        }
      }
    }
    const float sc = wsum > 0.f ? 1.f / wsum : 0.f;
    // row erow of the tile: 16-byte chunk j at j ^ (bits 7.. of its offset), as the
    // tensor map's swizzle of CW * 2 bytes places it
    constexpr uint32_t kSwzMask = CW * 2 / 16 - 1;
    const uint32_t tile = smem_u32(smem) + kOutOff;
#pragma unroll
    for (int j = 0; j < CW / 8; ++j) {
      const uint32_t off = erow * (CW * 2) + j * 16;
      st_shared_v4(tile + (off ^ (((off >> 7) & kSwzMask) << 4)),
                   pack_bf16(acc[8 * j] * sc, acc[8 * j + 1] * sc), pack_bf16(acc[8 * j + 2] * sc, acc[8 * j + 3] * sc),
                   pack_bf16(acc[8 * j + 4] * sc, acc[8 * j + 5] * sc), pack_bf16(acc[8 * j + 6] * sc, acc[8 * j + 7] * sc));
    }
    if (row_ok && split == 0 && p.lse_out) p.lse_out[orow] = wsum > 0.f ? mx + logf(wsum) : -INFINITY;
    fence_proxy_async_smem();
    asm volatile("bar.sync 1, 256;" ::: "memory");
    if (threadIdx.x == 0) {
      // rows past the last token are clipped by the tensor map
      tma_store_4d(&p.tm_out, tile, split * CW, ce.kvh * p.G, ce.rt * (kTcRows / p.G), ce.req);
      bulk_commit();
    }
  }
  cluster_sync_all();   // 2: every copy has landed; no CTA leaves while a peer may still read its slots
  if (threadIdx.x == 0) bulk_wait_read_all();   // the output tile has been read
}

// Epilogue of the softmax warps (warps 0..7, one CTA row per thread): O from
// tensor memory, normalised, written as bf16 -- directly, or after merging the
// split-KV chunks of the row tile.  A separate (not inlined) function, so that
// its registers do not press on the main loop's.
template <int D>
__device__ __noinline__ void tc_epilogue(const AttnParams& p, uint8_t* smem, uint32_t o_col, bool ok,
                                         float m_run, float l_run, int ntile) {
  using L = TcLayout<D>;
  const uint32_t sbase = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR_OFF);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 520);
  volatile int* last_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 524);
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int G = p.G;
  grid_dep_wait();   // before the first global write (the producer thread has waited already)
  const TcCta ce = tc_cta(p, blockIdx.x);
  const int nsplit = ce.nsplit;
  const int erow = threadIdx.x;                               // CTA row = thread (warps 0..7)
  const int epr = ce.rt * kTcRows + erow;                     // packed row
  const bool row_ok = epr / G < p.S;
  if (ok && ntile > 0) ok = warp_wait(bar(B_O), 0, abort_flag, p.wait_limit, p.status);
  if (ok) tc_fence_after();
  const float inv_l = (l_run > 0.f) ? 1.f / l_run : 0.f;
  const float lse = (ok && l_run > 0.f) ? (m_run + log2f(l_run)) * 0.69314718055994531f : -INFINITY;
  // output row of packed row `pr`: token pr / G, head kvh * G + pr % G
  auto out_row = [&](int pr) {
    return ((long long)ce.req * p.S + pr / G) * p.Hq + ce.kvh * G + pr % G;
  };
  if (p.work.cluster > 0) {
    if (nsplit == 4)
      tc_cluster_merge<D, 4>(p, smem, ce, o_col, ok, ntile, inv_l, lse, out_row(epr), row_ok);
    else
      tc_cluster_merge<D, 2>(p, smem, ce, o_col, ok, ntile, inv_l, lse, out_row(epr), row_ok);
  } else if (nsplit > 1) {
    // Independent splits: publish this chunk's normalised O and its
    // log-sum-exp through global memory; the last CTA of the (request, KV
    // head, row tile) to arrive merges all chunks.  A published piece is 32
    // columns of the 256 rows as fp16 pairs [16][256] (each row divided by the
    // power of 2 just above its largest magnitude in those columns), then the
    // 256 scales: half the bytes of fp32, and a warp's accesses to one pair
    // are 128 consecutive bytes.  The merge reads every chunk back, the
    // merging CTA's own too, so the sum is the same whichever CTA is last.
    const int cta = cta_index_fresh();
    const int r = erow;
    const long long orow = out_row(epr);
    const int req = ce.req, kvh = ce.kvh, rt = ce.rt;
    constexpr int kVals = 16 * kTcRows * 4;                 // 16 KiB of fp16 pairs
    constexpr int kPiece = kVals + kTcRows * 4;             // + 1 KiB of scales
    constexpr int kWtsOff = L::BAR_OFF - kMaxSplits * kTcRows * 4;   // merge weights [kMaxSplits][256]
    constexpr int kRing = (kWtsOff / kPiece) < 8 ? (kWtsOff / kPiece) : 8;
    static_assert(D / 32 * kPiece <= kWtsOff && kRing >= 2, "staging buffers");
    uint8_t* const part = reinterpret_cast<uint8_t*>(p.part_o);
    auto piece_of = [&](int c_idx, int c) { return part + ((long long)c_idx * (D / 32) + c) * kPiece; };
#pragma unroll 1
    for (int c = 0; c < D / 32; ++c) {
      float o[32];
      if (ok && ntile > 0) {
        tmem_ld32(o_col + c * 32, o);
        tc_wait_ld();
#pragma unroll
        for (int k = 0; k < 32; ++k) o[k] *= inv_l;
      } else {
#pragma unroll
        for (int k = 0; k < 32; ++k) o[k] = 0.f;
      }
      float amax = 0.f;
#pragma unroll
      for (int k = 0; k < 32; ++k) amax = fmaxf(amax, fabsf(o[k]));
      const int ex = (__float_as_int(amax) >> 23) & 0xff;
      const float scale = (amax > 0.f && ex < 254) ? __int_as_float((ex + 1) << 23) : 1.f;
      const float inv = 1.f / scale;
      uint32_t* dst = reinterpret_cast<uint32_t*>(smem + c * kPiece) + r;
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        const __half2 h = __floats2half2_rn(o[2 * k] * inv, o[2 * k + 1] * inv);
        dst[k * kTcRows] = *reinterpret_cast<const uint32_t*>(&h);
      }
      reinterpret_cast<float*>(smem + c * kPiece + kVals)[r] = scale;
    }
    p.part_lse[(long long)cta * kTcRows + r] = lse;
    fence_proxy_async_smem();
    asm volatile("bar.sync 1, 256;" ::: "memory");
    if (threadIdx.x == 0) {
      bulk_store(piece_of(cta, 0), sbase, (D / 32) * kPiece);
      bulk_commit();
      bulk_wait_all();
      fence_proxy_async_all();
    }
    // every CTA arrives, also after a timeout, so the count always completes;
    // the merge runs only without an abort (a warp whose wait failed raised
    // the flag before the barrier above), decided once for all warps
    __threadfence();
    asm volatile("bar.sync 1, 256;" ::: "memory");
    if (threadIdx.x == 0) {
      const int unit = (req * p.Hkv + kvh) * p.work.row_tiles + rt;
      const bool last = atomicAdd(&p.unit_cnt[unit], 1) == nsplit - 1;
      bool fits = nsplit <= kMaxSplits;   // merge weights: one buffer of kMaxSplits x 256
      if (last && !fits) set_status(p.status, ATTUNER_ERR_DEVICE_CHECK);
      *last_flag = (last && fits && !*abort_flag) ? 1 : 0;
    }
    asm volatile("bar.sync 1, 256;" ::: "memory");
    if (*last_flag) {
      __threadfence();
      fence_proxy_async_all();
      const int c0 = p.work.base[req] + kvh * p.work.row_tiles + rt;   // CTA of split 0
      const int cstride = p.Hkv * p.work.row_tiles;
      // merge weights exp(lse_s - max) of this row, one per split; the
      // splits' log-sum-exps are loaded together (one L2 round trip, not one
      // per split), eight at a time
      float* wt = reinterpret_cast<float*>(smem + kWtsOff);
      float mx = -INFINITY;
      for (int s0 = 0; s0 < nsplit; s0 += 8) {
        float ls[8];
#pragma unroll
        for (int i = 0; i < 8; ++i)
          ls[i] = (s0 + i < nsplit) ? __ldcg(p.part_lse + (long long)(c0 + (s0 + i) * cstride) * kTcRows + r) : -INFINITY;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          mx = fmaxf(mx, ls[i]);
          if (s0 + i < nsplit) wt[(s0 + i) * kTcRows + r] = ls[i];
        }
      }
      float wsum = 0.f;
      for (int sp = 0; sp < nsplit; ++sp) {
        const float ls = wt[sp * kTcRows + r];
        const float w = (ls == -INFINITY) ? 0.f : __expf(ls - mx);
        wsum += w;
        wt[sp * kTcRows + r] = w;
      }
      const float inv_w = wsum > 0.f ? 1.f / wsum : 0.f;
      // piece i = (column block i / nsplit, split i % nsplit) streams through the
      // ring of kRing buffers; warp 0 issues the copies
      const int n_pieces = (D / 32) * nsplit;
      auto issue = [&](int i) {
        const int b = i % kRing;
        mbar_expect_tx(bar(B_MF + b), kPiece);
        bulk_load(sbase + b * kPiece, piece_of(c0 + (i % nsplit) * cstride, i / nsplit), kPiece, bar(B_MF + b));
      };
      int issued = 0;
      if (warp == 0) {
        if (lane == 0)
          for (int i = 0; i < min(kRing, n_pieces); ++i) issue(i);
        issued = min(kRing, n_pieces);
      }
      asm volatile("bar.sync 1, 256;" ::: "memory");   // weights visible to all rows' threads
      bool mok = true;
#pragma unroll 1
      for (int c = 0; mok && c < D / 32; ++c) {
        float acc[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) acc[k] = 0.f;
#pragma unroll 1
        for (int sp = 0; sp < nsplit; ++sp) {
          const int i = c * nsplit + sp, b = i % kRing;
          if (!(mok = warp_wait(bar(B_MF + b), (i / kRing) & 1, abort_flag, p.wait_limit, p.status))) break;
          const uint8_t* pc = smem + b * kPiece;
          const float wk = wt[sp * kTcRows + r] * reinterpret_cast<const float*>(pc + kVals)[r];
          const uint32_t* src = reinterpret_cast<const uint32_t*>(pc) + r;
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const uint32_t bits = src[k * kTcRows];
            const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&bits));
            acc[2 * k] = __fmaf_rn(wk, f.x, acc[2 * k]);
            acc[2 * k + 1] = __fmaf_rn(wk, f.y, acc[2 * k + 1]);
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(bar(B_ME + b));
          if (warp == 0 && i + kRing < n_pieces) {
            if (!(mok = warp_wait(bar(B_ME + b), (i / kRing) & 1, abort_flag, p.wait_limit, p.status))) break;
            if (lane == 0) issue(i + kRing);
            ++issued;
          }
        }
        if (mok && row_ok) store_cols<D, 32>(p.out, orow, c * 32, acc, inv_w);
      }
      if (warp == 0 && !mok && lane == 0) {   // let the copies this CTA issued land
        for (int i = max(0, issued - kRing); i < issued; ++i)
          mbar_drain(bar(B_MF + i % kRing), (i / kRing) & 1, p.status);
      }
      if (mok && row_ok && p.lse_out) p.lse_out[orow] = wsum > 0.f ? mx + logf(wsum) : -INFINITY;
    }
  } else if (ok && ntile > 0) {
    const long long orow = out_row(epr);
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
      float o[32];
      tmem_ld32(o_col + c * 32, o);
      tc_wait_ld();
      if (row_ok) store_cols<D, 32>(p.out, orow, c * 32, o, inv_l);
    }
    if (row_ok && p.lse_out) p.lse_out[orow] = lse;
  }
}

// kLayout: some request of the plan has online spans before artifacts (the
// general visibility rule); false keeps the plain rule of the common layout.
template <int D, bool kLayout>
__global__ void __launch_bounds__(384, 1) attn_tc_kernel(const __grid_constant__ AttnParams p) {
  using L = TcLayout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR_OFF);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::BAR_OFF + 512);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 520);
  volatile int* last_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 524);
  int* list = reinterpret_cast<int*>(smem + L::LIST_OFF);
  auto bar = [&](int i) { return smem_u32(&bars[i]); };

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int G = p.G;

  // ---- which (request, kv head, row tile, split) this CTA owns
  const int cta = blockIdx.x;
  const TcCta cw = tc_cta(p, cta);
  const int req = cw.req, rt = cw.rt, kvh = cw.kvh;
  const int boff = p.plan.blk_off[req];
  const int nab = p.plan.blk_off[req + 1] - boff;
  const int nsuf = (p.S_kv + kBlockTokens - 1) / kBlockTokens;   // chunks of online rows
  const int row0 = rt * kTcRows;
  const int last_row = min(row0 + kTcRows - 1, p.S * G - 1);
  const int lim_last = (p.S_kv - p.S) + last_row / G;   // online row of the tile's last query
  // The row tile reads its own list of slots: the artifact slots its last
  // query sees (queries are in prompt order, so no query of the tile sees
  // more), then the online chunks up to the one holding that query's key.
  const int nart = kLayout ? art_slots_seen(p.plan, req, lim_last, nab) : nab;
  const int last_vis = nart + lim_last / kBlockTokens;
  int v_lo, v_hi;
  kv_part_range(p.kv_part, nart, nsuf, v_lo, v_hi);
  const int b0 = v_lo + cw.split * cw.chunk;
  const int b1 = min(min(b0 + cw.chunk, v_hi), last_vis + 1);
  const int nblk = max(0, b1 - b0);
  const int ntile = (nblk + 1) / 2;
  const int pool_rows = p.plan.pool_blocks * p.Hkv * kBlockTokens;
  // keys rotated at assembly: the K rows of this CTA's slot b0 + i
  const CUtensorMap* kslot = p.k_by_slot ? &p.tm_kslot : nullptr;
  auto kslot_row = [&](int i) { return ((boff + b0 + i) * p.Hkv + kvh) * kBlockTokens; };

  // ---- slots of this chunk: >0 artifact block, <0 online chunk, 0 none
  auto slot_entry = [&](int i) {
    int e = 0;
    if (i < nblk) {
      const int b = b0 + i;
      if (b < nart) {
        e = p.plan.blocks[boff + b];
        if (e <= 0 || (e >> 7) >= p.plan.pool_blocks || (e & 127) < 1 || (e & 127) > kBlockTokens) {
          set_status(p.status, ATTUNER_ERR_DEVICE_CHECK);
          e = 0;
        }
      } else {
        e = online_entry((b - nart) * kBlockTokens, kBlockTokens);
      }
    }
    return e;
  };
  constexpr uint32_t tile_bytes = 2 * L::NH * (kBlockTokens * 128);
  // The producer thread initialises the barriers and starts the first K tile
  // and Q before the block's first barrier, so their loads overlap the slot
  // list, the TMEM allocation and the first fetches of the other roles' code.
  if (warp == kProducerWarp && lane == 0) {
    for (int i = 0; i < B_COUNT; ++i)
      mbar_init(bar(i), (i == B_PF || i == B_PF + 1) ? 4u : (i >= B_ME ? 8u : 1u));
    *abort_flag = 0;
    fence_mbar_init();
    if (ntile > 0) {
      tma_prefetch_desc(&p.tm_q);
      tma_prefetch_desc(&p.tm_kpool);
      tma_prefetch_desc(&p.tm_vpool);
      const int e0 = slot_entry(0), e1 = slot_entry(1);
      // Only kernels that never signal an early launch write the paged pool,
      // so pool blocks may load while the previous kernel of the stream is
      // still running; Q and suffix K/V wait for it.
      if (e0 < 0 || e1 < 0) grid_dep_wait();
      const uint32_t kd = sbase + L::K_OFF;
      mbar_expect_tx(bar(B_KF), tile_bytes);
      load_slot<D>(kd, e0, &p.tm_kpool, &p.tm_ksuf, bar(B_KF), kvh, p.Hkv, req, pool_rows, kslot, kslot_row(0));
      load_slot<D>(kd + kBlockTokens * 128, e1, &p.tm_kpool, &p.tm_ksuf, bar(B_KF), kvh, p.Hkv, req, pool_rows,
                   kslot, kslot_row(1));
      grid_dep_wait();
      mbar_expect_tx(bar(B_Q), 2 * L::NH * L::HALF);
#pragma unroll
      for (int qt = 0; qt < 2; ++qt) {
#pragma unroll
        for (int h = 0; h < L::NH; ++h)
          tma_load_5d(sbase + L::Q_OFF + (qt * L::NH + h) * L::HALF, &p.tm_q, bar(B_Q), h * 64, 0, kvh,
                      (row0 + qt * kTcTileRows) / G, req);
      }
    }
  }
  for (int i = threadIdx.x; i < 2 * ntile; i += blockDim.x) list[i] = slot_entry(i);
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), L::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (warp >= 8) {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kCtrlRegs));
  if (warp == kProducerWarp) {
    // ================= TMA producer =================
    if (lane == 0 && ntile > 0) {
      // K0 and Q are in flight (issued before the block's first barrier)
      int issued_k = 1, issued_v = 0;
      for (int j = 0; j < ntile; ++j) {
        const int st = j % L::NS;
        const int e0 = list[2 * j], e1 = list[2 * j + 1];
        if (j > 0) {
          if (j >= L::NS &&
              !mbar_wait(bar(B_KE + st), ((j / L::NS) - 1) & 1, abort_flag, p.wait_limit, p.status))
            break;
          const uint32_t kd = sbase + L::K_OFF + st * L::NH * L::HALF;
          mbar_expect_tx(bar(B_KF + st), tile_bytes);
          load_slot<D>(kd, e0, &p.tm_kpool, &p.tm_ksuf, bar(B_KF + st), kvh, p.Hkv, req, pool_rows, kslot,
                       kslot_row(2 * j));
          load_slot<D>(kd + kBlockTokens * 128, e1, &p.tm_kpool, &p.tm_ksuf, bar(B_KF + st), kvh,
                       p.Hkv, req, pool_rows, kslot, kslot_row(2 * j + 1));
          issued_k = j + 1;
        }
        if (j >= L::NS &&
            !mbar_wait(bar(B_VE + st), ((j / L::NS) - 1) & 1, abort_flag, p.wait_limit, p.status))
          break;
        const uint32_t vd = sbase + L::V_OFF + st * L::NH * L::HALF;
        mbar_expect_tx(bar(B_VF + st), tile_bytes);
        load_slot<D>(vd, e0, &p.tm_vpool, &p.tm_vsuf, bar(B_VF + st), kvh, p.Hkv, req, pool_rows);
        load_slot<D>(vd + kBlockTokens * 128, e1, &p.tm_vpool, &p.tm_vsuf, bar(B_VF + st), kvh,
                     p.Hkv, req, pool_rows);
        issued_v = j + 1;
      }
      if (*abort_flag) {   // let every copy this CTA issued land before exiting
        mbar_drain(bar(B_Q), 0, p.status);
        for (int j = (issued_k > L::NS ? issued_k - L::NS : 0); j < issued_k; ++j)
          mbar_drain(bar(B_KF + j % L::NS), (j / L::NS) & 1, p.status);
        for (int j = (issued_v > L::NS ? issued_v - L::NS : 0); j < issued_v; ++j)
          mbar_drain(bar(B_VF + j % L::NS), (j / L::NS) & 1, p.status);
      }
    }
  } else if (warp == kMmaWarp) {
    // ================= MMA issuer (one thread) =================
    if (lane == 0 && ntile > 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(128, 128, 0, 0);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, 0, 1);
      bool any = false;
      auto wait = [&](int b, uint32_t par) { return mbar_wait(bar(b), par, abort_flag, p.wait_limit, p.status); };
      auto issue_qk = [&](int qt, int st) {
        const uint32_t q_s = sbase + L::Q_OFF + qt * L::NH * L::HALF;
        const uint32_t k_s = sbase + L::K_OFF + st * L::NH * L::HALF;
#pragma unroll
        for (int k = 0; k < D / 16; ++k) {
          const uint32_t off = (k / 4) * L::HALF + (k % 4) * 32;
          umma_bf16(tmem + s_col_of(qt), sdesc_sw128(q_s + off, 16, 1024), sdesc_sw128(k_s + off, 16, 1024),
                    idesc_qk, k > 0 ? 1u : 0u);
        }
        umma_commit(bar(B_SF + qt));
        any = true;
      };
      auto issue_pv = [&](int qt, int st, int j) {
        const uint32_t v_s = sbase + L::V_OFF + st * L::NH * L::HALF;
#pragma unroll
        for (int k = 0; k < 8; ++k)
          umma_bf16_ts(tmem + o_col_of(qt), tmem + s_col_of(qt) + k * 8,
                       sdesc_sw128(v_s + k * 2048, L::HALF, 1024), idesc_pv, (j > 0 || k > 0) ? 1u : 0u);
      };
      bool ok = wait(B_Q, 0) && wait(B_KF, 0);
      if (ok) {
        tc_fence_after();
        issue_qk(0, 0);
        issue_qk(1, 0);
        umma_commit(bar(B_KE));
      }
      for (int j = 0; ok && j < ntile; ++j) {
        const int st = j % L::NS, st1 = (j + 1) % L::NS;
        const bool more = j + 1 < ntile;
        if (!(ok = wait(B_PF, j & 1) && wait(B_VF + st, (j / L::NS) & 1))) break;
        tc_fence_after();
        issue_pv(0, st, j);
        if (more) {
          if (!(ok = wait(B_KF + st1, ((j + 1) / L::NS) & 1))) break;
          tc_fence_after();
          issue_qk(0, st1);
        }
        if (!(ok = wait(B_PF + 1, j & 1))) break;
        tc_fence_after();
        issue_pv(1, st, j);
        umma_commit(bar(B_VE + st));
        if (more) {
          issue_qk(1, st1);
          umma_commit(bar(B_KE + st1));
        }
      }
      if (ok) {
        umma_commit(bar(B_O));
      } else if (any) {
        umma_commit(bar(B_DRAIN));
        mbar_drain(bar(B_DRAIN), 0, p.status);
      }
    }
  }
  // cluster mode: the softmax warps' two cluster barriers count every thread
  if (p.work.cluster > 0) {
    cluster_sync_all();
    cluster_sync_all();
  }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kSoftRegs));
    // ================= softmax + epilogue: warps 0..3 -> Q0, 4..7 -> Q1 =================
    const int qt = warp / 4;
    const int quad = warp & 3;
    const int r = qt * kTcTileRows + quad * 32 + lane;   // CTA row
    const int pr = row0 + r;                             // packed row
    const int tok = pr / G;
    // What this query (online row lim) sees: online keys up to its own online
    // row (online rows are in assembled order) and, with online spans before
    // artifacts, only the artifact slots before its span (vs, chunk-relative).
    const int lim = (p.S_kv - p.S) + tok;
    const int vs = kLayout ? art_slots_seen(p.plan, req, lim, nab) - b0 : 0;
    auto visible = [&](int s, int e) {
      if (e > 0) return (kLayout && s >= vs) ? 0 : (e & 127);
      if (e < 0) return min(max(lim - slot_row0(e) + 1, 0), kBlockTokens);
      return 0;
    };
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    const uint32_t s_col = tmem + lane_base + s_col_of(qt);
    const uint32_t o_col = tmem + lane_base + o_col_of(qt);
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    if (p.inject_stuck && warp == 2)
      ok = warp_wait(bar(B_NEVER), 0, abort_flag, p.wait_limit, p.status);   // nothing arrives: times out
    for (int j = 0; ok && j < ntile; ++j) {
      if (!warp_wait(bar(B_SF + qt), j & 1, abort_flag, p.wait_limit, p.status)) { ok = false; break; }
      tc_fence_after();
      float sc[128];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(s_col + c * 32, sc + c * 32);
      // while the TMEM loads are in flight: visible keys of the two slots, and
      // one warp vote (most tiles are fully visible and skip the masking code)
      const int nv0 = visible(2 * j, list[2 * j]), nv1 = visible(2 * j + 1, list[2 * j + 1]);
      const bool need_mask = __any_sync(0xffffffffu, min(nv0, nv1) < kBlockTokens);
      tc_wait_ld();
      if (need_mask) {
        mask_tail(sc, nv0);
        mask_tail(sc + 64, nv1);
      }
      // row max: eight independent chains of 3-input max, then a small tree
      float mk[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) mk[k] = fmaxf(sc[k], sc[k + 8]);
#pragma unroll
      for (int c = 16; c < 128; c += 16) {
#pragma unroll
        for (int k = 0; k < 8; ++k) mk[k] = fmax3(mk[k], sc[c + k], sc[c + k + 8]);
      }
      float mx = fmax3(fmax3(mk[0], mk[1], mk[2]), fmax3(mk[3], mk[4], mk[5]), fmaxf(mk[6], mk[7]));
      mx *= p.scale_log2;
      float alpha = 1.f;
      if (mx > m_run + 8.f) {              // move the reference max only when it grows past 2^8
        alpha = ex2(m_run - mx);           // m_run = -inf gives 0
        m_run = mx;
      }
      const float neg = (m_run == -INFINITY) ? 0.f : -m_run;
      // p = 2^(s * log2(e)/sqrt(d) - m): packed fp32 FMA, then ex2; row sum in packed chains
      const uint64_t sc2 = f2_pack(p.scale_log2, p.scale_log2), ng2 = f2_pack(neg, neg);
      uint64_t acc2[4] = {0ull, 0ull, 0ull, 0ull};
      // P as bf16 pairs (key k in column k/2) over the first 64 columns of this
      // tile's S region; the first half is stored while the second is computed
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        uint32_t pk[32];
#pragma unroll
        for (int c = 64 * h; c < 64 * h + 64; c += 2) {
          float x0, x1;
          f2_unpack(f2_fma(f2_pack(sc[c], sc[c + 1]), sc2, ng2), x0, x1);
          x0 = ex2(x0);
          x1 = ex2(x1);
          acc2[(c >> 1) & 3] = f2_add(acc2[(c >> 1) & 3], f2_pack(x0, x1));
          pk[(c >> 1) & 31] = pack_bf16(x0, x1);
        }
        tmem_st32(s_col + 32 * h, reinterpret_cast<const float*>(pk));
      }
      {
        float a0, a1;
        f2_unpack(f2_add(f2_add(acc2[0], acc2[1]), f2_add(acc2[2], acc2[3])), a0, a1);
        l_run = l_run * alpha + (a0 + a1);
      }
      // O is current here (the commit that signalled S also covers the previous PV)
      if (j >= 1 && __any_sync(0xffffffffu, alpha != 1.f)) {
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          float o[32];
          tmem_ld32(o_col + c * 32, o);
          tc_wait_ld();
#pragma unroll
          for (int k = 0; k < 32; ++k) o[k] *= alpha;
          tmem_st32(o_col + c * 32, o);
        }
      }
      tc_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(B_PF + qt));
    }

    tc_epilogue<D>(p, smem, o_col, ok, m_run, l_run, ntile);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, L::TMEM_COLS);
  }
}

template <int D, bool kLayout>
static cudaError_t launch_attn_tc_t(const AttnParams& p, cudaStream_t st) {
  using L = TcLayout<D>;
  // setmaxnreg.inc waits until the registers it asks for are free in the
  // block's launch budget: never launch a split that exceeds that budget.
  // (checked once per instantiation: the register count is fixed at build time)
  static const cudaError_t regs = [] {
    cudaFuncAttributes fa{};
    const cudaError_t r = cudaFuncGetAttributes(&fa, attn_tc_kernel<D, kLayout>);
    if (r != cudaSuccess) return r;
    return fa.numRegs * 384 < 128 * kCtrlRegs + 256 * kSoftRegs ? cudaErrorLaunchOutOfResources : cudaSuccess;
  }();
  if (regs != cudaSuccess) return regs;
  cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<D, kLayout>, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM);
  if (e != cudaSuccess) return e;
  return launch_pdl(attn_tc_kernel<D, kLayout>, dim3(p.work.n_cta), dim3(384), (size_t)L::SMEM, st, p.work.cluster, p);
}

// clusters of `ns` CTAs of this kernel that fit on the device at once (0: none)
template <int D>
static int attn_tc_max_clusters_t(int ns) {
  using L = TcLayout<D>;
  if (cudaFuncSetAttribute(attn_tc_kernel<D, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(ns);
  cfg.blockDim = dim3(384);
  cfg.dynamicSmemBytes = L::SMEM;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = ns;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, attn_tc_kernel<D, false>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

int attn_tc_max_clusters(int D, int ns) {
  if (D == 128) return attn_tc_max_clusters_t<128>(ns);
  if (D == 64) return attn_tc_max_clusters_t<64>(ns);
  return 0;
}

cudaError_t launch_attn_tc(const AttnParams& p, int D, cudaStream_t st) {
  const bool layout = p.plan.has_spans != 0;
  if (D == 128) return layout ? launch_attn_tc_t<128, true>(p, st) : launch_attn_tc_t<128, false>(p, st);
  if (D == 64) return layout ? launch_attn_tc_t<64, true>(p, st) : launch_attn_tc_t<64, false>(p, st);
  return cudaErrorInvalidValue;
}

}  // namespace att
