// attn_mma.cu - K3: split-KV attention for few query rows per (request, KV
// head), the decode step of Sec. 3 (generated tokens read the frozen
// artifact KV plus the online KV through the adapted query) and, as a
// second kernel for any S, the same attention as attn_tc.cu, with K4, the
// log-sum-exp merge of its split-KV chunks, done by the last CTA of each row
// tile to finish; and APE's calibrated combination of two partial results.
//
// K3 streams K/V: every (request, KV head) reads its assembled K/V once
// (4 KiB per token at Hkv = 8, d = 128).  One CTA owns 16 packed query rows
// (token * G + head_in_group) of one request and KV head, and one chunk of its
// virtual block list; the CTAs launch KV-head-major, so requests that share
// an artifact read its blocks from L2 after the first.  With shared reads
// (kShare) the 16 rows are those of up to 16 / (S G) requests that use the
// same artifact: a CTA reads one chunk of that artifact once for all of them
// (or one chunk of a single request's online rows), and every request's
// partial results - one per chunk of each artifact it lists, one per online
// chunk - are merged by the last CTA to finish one of them.  Warp 4 streams
// 64-token K/V blocks with TMA (128-byte swizzle) into a ring of 3 stages
// (2 with shared reads; two or three CTAs share an SM, so one's prologue and
// merge overlap the others' loads); warps
// 0..3 each take 16 of the 64 keys of every block (intra-CTA split over
// keys), run QK^T and PV with m16n8k16 warp MMAs (tensor work is ~5% of the
// memory time here), keep an online softmax in registers, and merge their
// partial results through shared memory at the end.
#include <math.h>

#include "kernels.h"

namespace att {

// Per-request reads: a 3-stage ring, two CTAs per SM.  Shared reads: a
// 2-stage ring, three CTAs per SM (their CTAs are shorter, so a third CTA's
// loads cover more of the others' prologues and merges: 0.210 against 0.213 ms
// on the 64-request decode step, where the per-request kernel took 0.310
// against 0.285 ms in that shape).
template <int D, bool kShare>
struct MmaLayout {
  static constexpr int CTAS = kShare ? 3 : 2;        // resident CTAs per SM
  static constexpr int NH = D / 64;
  static constexpr int NS = kShare ? 2 : 3;
  static constexpr int BLK = kBlockTokens * 128;      // one 64-row x 128 B box
  static constexpr int STAGE = 2 * NH * BLK;          // K halves then V halves
  static constexpr int BAR_OFF = NS * STAGE;
  static constexpr int LIST_OFF = BAR_OFF + 256;
  static constexpr int MEM_OFF = LIST_OFF + kMmaMaxChunkBlocks * 4;   // shared reads: [16][4] member table
  static constexpr int MERGE_BYTES = 4 * 16 * (D + 2) * 4;   // per warp: O[16][D], m[16], l[16]
  static constexpr int SMEM = MEM_OFF + 16 * 16 + 1024;   // CTAS of them fit in an SM's shared memory
  static_assert(MERGE_BYTES <= BAR_OFF, "merge area aliases the stage ring");
};

// The merge of n partial results of one query row (K4): record k of the row
// at part_lse[rec(k)] and part_o[rec(k) * D ...], in order k = 0 .. n - 1:
// lse = log sum_k exp(lse_k),  O = sum_k exp(lse_k - lse) O_k.  The calling
// thread writes its CPT = D / 8 columns from c0 of output row orow.  The
// loads of eight log-sum-exps, then of two records, are issued before any is
// used: the merge is bound by L2 latency, not by its few bytes (two records
// and not four keep the three-CTAs-per-SM kernel within its registers).
template <int D, class Rec>
ATT_DEV void merge_records(const AttnParams& p, int n, Rec rec, int c0, long long orow, int tid) {
  constexpr int CPT = D / 8, NV = CPT / 4;
  float Ms = -INFINITY;
  int k = 0;
  for (; k + 8 <= n; k += 8) {
    float l[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) l[i] = __ldcg(p.part_lse + rec(k + i));
#pragma unroll
    for (int i = 0; i < 8; ++i) Ms = fmaxf(Ms, l[i]);
  }
  for (; k < n; ++k) Ms = fmaxf(Ms, __ldcg(p.part_lse + rec(k)));
  float W = 0.f;
  float acc[CPT];
#pragma unroll
  for (int c = 0; c < CPT; ++c) acc[c] = 0.f;
  auto add = [&](float ls, const float4* v) {
    const float w = (ls == -INFINITY) ? 0.f : __expf(ls - Ms);
    W += w;
#pragma unroll
    for (int c = 0; c < NV; ++c) {
      acc[4 * c] += w * v[c].x; acc[4 * c + 1] += w * v[c].y; acc[4 * c + 2] += w * v[c].z; acc[4 * c + 3] += w * v[c].w;
    }
  };
  k = 0;
  for (; k + 2 <= n; k += 2) {
    float ls[2];
    float4 v[2][NV];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const long long at = rec(k + i);
      ls[i] = __ldcg(p.part_lse + at);
#pragma unroll
      for (int c = 0; c < NV; ++c) v[i][c] = __ldcg(reinterpret_cast<const float4*>(p.part_o + at * D + c0) + c);
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) add(ls[i], v[i]);
  }
  for (; k < n; ++k) {
    const long long at = rec(k);
    float4 v[NV];
#pragma unroll
    for (int c = 0; c < NV; ++c) v[c] = __ldcg(reinterpret_cast<const float4*>(p.part_o + at * D + c0) + c);
    add(__ldcg(p.part_lse + at), v);
  }
  const float invW = (W > 0.f) ? 1.f / W : 0.f;
  uint4* dst = reinterpret_cast<uint4*>(p.out + orow * D + c0);
#pragma unroll
  for (int c = 0; c < CPT; c += 8)
    dst[c / 8] = make_uint4(pack_bf16(acc[c] * invW, acc[c + 1] * invW), pack_bf16(acc[c + 2] * invW, acc[c + 3] * invW),
                            pack_bf16(acc[c + 4] * invW, acc[c + 5] * invW), pack_bf16(acc[c + 6] * invW, acc[c + 7] * invW));
  if ((tid & 7) == 0 && p.lse_out) p.lse_out[orow] = (W > 0.f) ? Ms + logf(W) : -INFINITY;
}

// kLayout: some request has online spans before artifacts (general visibility rule)
// kShare: the shared-read decomposition (WorkTable): a CTA reads one chunk of
// an artifact for the requests of one group of its references, or one chunk
// of a request's online rows, and every request's partials are merged by the
// last CTA to finish one of them
template <int D, bool kLayout, bool kShare>
__global__ void __launch_bounds__(160, kShare ? 3 : 2) attn_mma_kernel(const __grid_constant__ AttnParams p) {
  using L = MmaLayout<D, kShare>;
  static_assert(L::CTAS == (kShare ? 3 : 2), "launch bounds and layout agree");
  grid_dep_wait();     // Q and the suffix K/V may come from the previous kernel
  constexpr int NT = D / 8;           // n8 tiles of the output
  constexpr int KS = D / 16;          // k16 steps of QK^T
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR_OFF);   // full[NS], empty[NS], never
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 8 * (2 * L::NS + 1));
  int* list = reinterpret_cast<int*>(smem + L::LIST_OFF);
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  const int B_FULL = 0, B_EMPTY = L::NS, B_NEVER = 2 * L::NS;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int G = p.G;
  const int SG = p.S * G;                 // packed rows of one request
  int* mem = reinterpret_cast<int*>(smem + L::MEM_OFF);   // shared reads: request, partial, partials, last
  int kvh, req, row0, nblk, b0 = 0, boff = 0, nab = 0, cta = 0, nsplit = 1, rt = 0, n_mem = 1;
  if constexpr (kShare) {
    // Launch order: the artifact units KV-head-major (the CTAs resident at any
    // one time read one head's blocks), then every head's online-row units,
    // short CTAs that fill the grid's last wave.
    const int art_ctas = p.work.art_units * p.Hkv;
    int u;
    if ((int)blockIdx.x < art_ctas) {
      kvh = blockIdx.x / p.work.art_units;
      u = blockIdx.x % p.work.art_units;
    } else {
      const int v = blockIdx.x - art_ctas, per = p.work.n_req * p.work.suf_chunks;
      kvh = v / per;
      u = p.work.art_units + v % per;
    }
    const int C = p.work.chunk_blocks;
    row0 = 0;
    int chunk, src = 0, m_beg = 0;
    const bool art = u < p.work.art_units;
    if (art) {
      int lo = 0, hi = p.work.n_dist - 1;   // distinct artifact d: nsplit[d] <= u < nsplit[d + 1]
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.work.nsplit[mid] <= u) lo = mid; else hi = mid - 1;
      }
      const int r_beg = p.plan.dist_off[lo], r_end = p.plan.dist_off[lo + 1];
      const int nb = p.plan.dist_nb[lo];
      const int nch = (nb + C - 1) / C;
      const int local = u - p.work.nsplit[lo];
      chunk = local % nch;
      m_beg = r_beg + (local / nch) * p.work.members;
      n_mem = min(p.work.members, r_end - m_beg);
      req = p.plan.dref_req[m_beg];
      src = p.plan.dist_src[lo] + chunk * C;
      nblk = min(C, nb - chunk * C);
    } else {
      const int v = u - p.work.art_units;
      req = v / p.work.suf_chunks;
      chunk = v % p.work.suf_chunks;
      const int nsuf = (p.S_kv + kBlockTokens - 1) / kBlockTokens;
      nblk = min(C, nsuf - chunk * C);
    }
    for (int i = threadIdx.x; i < nblk; i += blockDim.x) {
      int e;
      if (art) {
        e = p.plan.blocks[src + i];
        if (e <= 0 || (e >> 7) >= p.plan.pool_blocks || (e & 127) < 1 || (e & 127) > kBlockTokens) {
          set_status(p.status, ATTUNER_ERR_DEVICE_CHECK);
          e = 0;
        }
      } else {
        e = online_entry((chunk * C + i) * kBlockTokens, kBlockTokens);
      }
      list[i] = e;
    }
    if (threadIdx.x < n_mem) {
      // the member's request, the index of this chunk among the request's
      // partials (its references' chunks in prompt order, then the suffix
      // chunks) and their count
      int r, j, nref;
      if (art) {
        r = p.plan.dref_req[m_beg + threadIdx.x];
        j = p.plan.dref_j[m_beg + threadIdx.x];
        nref = p.plan.dref_nref[m_beg + threadIdx.x];
      } else {
        r = req;
        j = 0;
        nref = p.plan.req_art_off[r + 1] - p.plan.req_art_off[r];
      }
      int k = j, P = nref;   // every reference one chunk
      if (!p.work.whole_refs) {
        k = 0;
        P = 0;
        const int i0 = p.plan.req_art_off[r];
        for (int i = 0; i < nref; ++i) {
          const int n = (p.plan.ref_nblk[i0 + i] + C - 1) / C;
          if (i < j) k += n;
          P += n;
        }
      }
      mem[4 * threadIdx.x + 0] = r;
      mem[4 * threadIdx.x + 1] = art ? k + chunk : P + chunk;
      mem[4 * threadIdx.x + 2] = P + p.work.suf_chunks;
      mem[4 * threadIdx.x + 3] = 0;
    }
  } else {
    // Launch order: KV head outermost, then request, split and row tile.  The
    // CTAs resident at any one time read the blocks of one KV head (about an
    // eighth of the pool), so requests that share an artifact find most of its
    // blocks still in L2.  `cta` is the request-major index that numbers the
    // split partials and the merge (base[r] + (split * Hkv + kvh) * row_tiles + rt).
    const int per_head = p.work.n_cta / p.Hkv;
    kvh = blockIdx.x / per_head;
    const int in_head = blockIdx.x % per_head;
    req = 0;
    {
      int lo = 0, hi = p.work.n_req - 1;   // the per-head bases are base[r] / Hkv
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.work.base[mid] / p.Hkv <= in_head) lo = mid; else hi = mid - 1;
      }
      req = lo;
    }
    const int rel = in_head - p.work.base[req] / p.Hkv;
    rt = rel % p.work.row_tiles;
    const int split = rel / p.work.row_tiles;
    cta = p.work.base[req] + (split * p.Hkv + kvh) * p.work.row_tiles + rt;
    nsplit = p.work.nsplit[req];
    boff = p.plan.blk_off[req];
    nab = p.plan.blk_off[req + 1] - boff;
    const int nsuf = (p.S_kv + kBlockTokens - 1) / kBlockTokens;   // chunks of online rows
    row0 = rt * kMmaRows;
    const int last_row = min(row0 + kMmaRows - 1, SG - 1);
    const int lim_last = (p.S_kv - p.S) + last_row / G;   // online row of the tile's last query
    // The row tile reads its own list of slots: the artifact slots its last
    // query sees (queries are in prompt order, so no query of the tile sees
    // more), then the online chunks up to the one holding that query's key.
    const int nart = kLayout ? art_slots_seen(p.plan, req, lim_last, nab) : nab;
    const int last_vis = nart + lim_last / kBlockTokens;
    int v_lo, v_hi;
    kv_part_range(p.kv_part, nart, nsuf, v_lo, v_hi);
    b0 = v_lo + split * p.work.chunk_blocks;
    const int b1 = min(min(b0 + p.work.chunk_blocks, v_hi), last_vis + 1);
    nblk = max(0, b1 - b0);

    for (int i = threadIdx.x; i < nblk; i += blockDim.x) {
      const int b = b0 + i;
      int e;
      if (b < nart) {
        e = p.plan.blocks[boff + b];
        if (e <= 0 || (e >> 7) >= p.plan.pool_blocks || (e & 127) < 1 || (e & 127) > kBlockTokens) {
          set_status(p.status, ATTUNER_ERR_DEVICE_CHECK);
          e = 0;
        }
      } else {
        e = online_entry((b - nart) * kBlockTokens, kBlockTokens);
      }
      list[i] = e;
    }
  }
  if (threadIdx.x == 0) {
    for (int i = 0; i < L::NS; ++i) {
      mbar_init(bar(B_FULL + i), 1);
      mbar_init(bar(B_EMPTY + i), 4);
    }
    mbar_init(bar(B_NEVER), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == 4) {
    // ================= TMA producer =================
    if (lane == 0) {
      const int pool_rows = p.plan.pool_blocks * p.Hkv * kBlockTokens;
      int issued = 0;
      for (int j = 0; j < nblk; ++j) {
        const int st = j % L::NS;
        if (j >= L::NS &&
            !mbar_wait(bar(B_EMPTY + st), ((j / L::NS) - 1) & 1, abort_flag, p.wait_limit, p.status))
          break;
        const uint32_t dst = sbase + st * L::STAGE;
        const uint32_t fb = bar(B_FULL + st);
        mbar_expect_tx(fb, L::STAGE);
        const int e = list[j];
#pragma unroll
        for (int h = 0; h < L::NH; ++h) {
          if (e < 0) {
            const int c = slot_row0(e);
            tma_load_4d(dst + h * L::BLK, &p.tm_ksuf, fb, h * 64, kvh, c, req);
            tma_load_4d(dst + (L::NH + h) * L::BLK, &p.tm_vsuf, fb, h * 64, kvh, c, req);
          } else {
            const int row = (e == 0) ? pool_rows : ((e >> 7) * p.Hkv + kvh) * kBlockTokens;
            if (e != 0 && p.k_by_slot)   // keys rotated at assembly, by the plan's slot index
              tma_load_2d(dst + h * L::BLK, &p.tm_kslot, fb, h * 64, ((boff + b0 + j) * p.Hkv + kvh) * kBlockTokens);
            else
              tma_load_2d(dst + h * L::BLK, &p.tm_kpool, fb, h * 64, row);
            tma_load_2d(dst + (L::NH + h) * L::BLK, &p.tm_vpool, fb, h * 64, row);
          }
        }
        issued = j + 1;
      }
      if (*abort_flag) {
        for (int j = (issued > L::NS ? issued - L::NS : 0); j < issued; ++j)
          mbar_drain(bar(B_FULL + j % L::NS), (j / L::NS) & 1, p.status);
      }
    }
    return;   // the producer takes no part in the merge below
  }

  // ================= consumers: warps 0..3 =================
  const int g = lane >> 2, t = lane & 3;
  // Q fragments of rows g and g+8 (A operand of m16n8k16, row-major)
  uint32_t qa[KS][4];
  int tok_r[2];
  long long qrow[2];
#pragma unroll
  for (int hr = 0; hr < 2; ++hr) {
    const int pr = row0 + g + 8 * hr;
    if constexpr (kShare) {   // member pr / SG, its packed row pr % SG
      const int mi = pr / SG, wr = pr % SG;
      tok_r[hr] = wr / G;
      qrow[hr] = (mi < n_mem) ? (((long long)mem[4 * mi] * p.S + tok_r[hr]) * p.Hq + kvh * G + wr % G) : -1;
    } else {
      tok_r[hr] = pr / G;
      qrow[hr] = (tok_r[hr] < p.S) ? (((long long)req * p.S + tok_r[hr]) * p.Hq + kvh * G + pr % G) : -1;
    }
  }
#pragma unroll
  for (int ks = 0; ks < KS; ++ks) {
#pragma unroll
    for (int hr = 0; hr < 2; ++hr) {
#pragma unroll
      for (int kh = 0; kh < 2; ++kh) {
        uint32_t v = 0;
        if (qrow[hr] >= 0)
          v = *reinterpret_cast<const uint32_t*>(p.q + qrow[hr] * D + ks * 16 + kh * 8 + 2 * t);
        qa[ks][hr + 2 * kh] = v;
      }
    }
  }
  // the thread's two query rows: online rows lim0 / lim1; with online spans
  // before artifacts, also the artifact slots they see, vs0 / vs1
  // (chunk-relative)
  const int lim0 = (p.S_kv - p.S) + tok_r[0];
  const int lim1 = (p.S_kv - p.S) + tok_r[1];
  const int vs0 = kLayout ? art_slots_seen(p.plan, req, (p.S_kv - p.S) + min(tok_r[0], p.S - 1), nab) - b0 : 0;
  const int vs1 = kLayout ? art_slots_seen(p.plan, req, (p.S_kv - p.S) + min(tok_r[1], p.S - 1), nab) - b0 : 0;

  float o[NT][4];
#pragma unroll
  for (int n = 0; n < NT; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  float m_r[2] = {-INFINITY, -INFINITY}, l_r[2] = {0.f, 0.f};
  bool ok = true;
  if (p.inject_stuck && warp == 0)
    ok = warp_wait(bar(B_NEVER), 0, abort_flag, p.wait_limit, p.status);   // nothing arrives: times out

  for (int j = 0; ok && j < nblk; ++j) {
    const int st = j % L::NS;
    if (!warp_wait(bar(B_FULL + st), (j / L::NS) & 1, abort_flag, p.wait_limit, p.status)) { ok = false; break; }
    const uint32_t ks_base = sbase + st * L::STAGE;
    const uint32_t vs_base = ks_base + L::NH * L::BLK;
    // ---- S = Q K^T for keys 16*warp .. +15 (two n8 tiles)
    float s[2][4];
#pragma unroll
    for (int n = 0; n < 2; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
    {
      const int mi = lane >> 3, ri = lane & 7;
      const int key = 16 * warp + 8 * (mi >> 1) + ri;
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        const int chunk = 2 * ks + (mi & 1);
        uint32_t b0r, b1r, b2r, b3r;
        ldmatrix_x4(ks_base + (chunk >> 3) * L::BLK + sw128_off(key, chunk & 7), b0r, b1r, b2r, b3r);
        mma_16816(s[0], qa[ks], b0r, b1r);
        mma_16816(s[1], qa[ks], b2r, b3r);
      }
    }
    // ---- mask
    const int e = list[j];
#pragma unroll
    for (int n = 0; n < 2; ++n) {
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int kb = 16 * warp + 8 * n + 2 * t + (c & 1);
        bool vis;
        if (e > 0) vis = kb < (e & 127) && (!kLayout || j < ((c < 2) ? vs0 : vs1));
        else if (e < 0) vis = (slot_row0(e) + kb) <= ((c < 2) ? lim0 : lim1);
        else vis = false;
        if (!vis) s[n][c] = -INFINITY;
      }
    }
    // ---- online softmax (rows g: c = 0,1; row g+8: c = 2,3)
    float alpha[2];
#pragma unroll
    for (int hr = 0; hr < 2; ++hr) {
      float mx = fmaxf(fmaxf(s[0][2 * hr], s[0][2 * hr + 1]), fmaxf(s[1][2 * hr], s[1][2 * hr + 1]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      mx *= p.scale_log2;
      const float m_new = fmaxf(m_r[hr], mx);
      const float m_use = (m_new == -INFINITY) ? 0.f : m_new;
      alpha[hr] = ex2(m_r[hr] - m_use);
      m_r[hr] = m_new;
      float rs = 0.f;
#pragma unroll
      for (int n = 0; n < 2; ++n) {
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const float pv = ex2(fmaf(s[n][2 * hr + c], p.scale_log2, -m_use));
          s[n][2 * hr + c] = pv;
          rs += pv;
        }
      }
      l_r[hr] = l_r[hr] * alpha[hr] + rs;
    }
#pragma unroll
    for (int n = 0; n < NT; ++n) {
      o[n][0] *= alpha[0]; o[n][1] *= alpha[0];
      o[n][2] *= alpha[1]; o[n][3] *= alpha[1];
    }
    // ---- O += P V (A = P from the S fragments; B = V via ldmatrix.trans)
    uint32_t pa[4];
    pa[0] = pack_bf16(s[0][0], s[0][1]);
    pa[1] = pack_bf16(s[0][2], s[0][3]);
    pa[2] = pack_bf16(s[1][0], s[1][1]);
    pa[3] = pack_bf16(s[1][2], s[1][3]);
    {
      const int mi = lane >> 3, ri = lane & 7;
      const int key = 16 * warp + ri + 8 * (mi & 1);
#pragma unroll
      for (int np = 0; np < NT / 2; ++np) {
        const int chunk = 2 * np + (mi >> 1);
        uint32_t b0r, b1r, b2r, b3r;
        ldmatrix_x4_trans(vs_base + (chunk >> 3) * L::BLK + sw128_off(key, chunk & 7), b0r, b1r, b2r, b3r);
        mma_16816(o[2 * np], pa, b0r, b1r);
        mma_16816(o[2 * np + 1], pa, b2r, b3r);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(bar(B_EMPTY + st));
  }

  // ---- merge the four warps (the stage ring is reused once every warp is done)
  asm volatile("bar.sync 1, 128;" ::: "memory");
  if (*abort_flag) return;
#pragma unroll
  for (int hr = 0; hr < 2; ++hr) {
    l_r[hr] += __shfl_xor_sync(0xffffffffu, l_r[hr], 1);
    l_r[hr] += __shfl_xor_sync(0xffffffffu, l_r[hr], 2);
  }
  float* mo = reinterpret_cast<float*>(smem) + warp * 16 * (D + 2);
#pragma unroll
  for (int n = 0; n < NT; ++n) {
    *reinterpret_cast<float2*>(mo + g * (D + 2) + 8 * n + 2 * t) = make_float2(o[n][0], o[n][1]);
    *reinterpret_cast<float2*>(mo + (g + 8) * (D + 2) + 8 * n + 2 * t) = make_float2(o[n][2], o[n][3]);
  }
  if (t == 0) {
    mo[g * (D + 2) + D] = m_r[0];
    mo[g * (D + 2) + D + 1] = l_r[0];
    mo[(g + 8) * (D + 2) + D] = m_r[1];
    mo[(g + 8) * (D + 2) + D + 1] = l_r[1];
  }
  asm volatile("bar.sync 1, 128;" ::: "memory");
  const float* mb = reinterpret_cast<const float*>(smem);
  const int tid = threadIdx.x;
  constexpr int CPT = D / 8;                    // columns per thread: 16 rows x 8 threads
  const int row = tid >> 3, c0 = (tid & 7) * CPT;
  float mw[4], lw[4];
  float M = -INFINITY;
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    mw[w] = mb[(w * 16 + row) * (D + 2) + D];
    lw[w] = mb[(w * 16 + row) * (D + 2) + D + 1];
    M = fmaxf(M, mw[w]);
  }
  const float Mu = (M == -INFINITY) ? 0.f : M;
  float wsum = 0.f, wt[4];
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    wt[w] = ex2(mw[w] - Mu);
    wsum += wt[w] * lw[w];
  }
  const float inv = (wsum > 0.f) ? 1.f / wsum : 0.f;
  const float lse = (wsum > 0.f) ? (Mu + log2f(wsum)) * 0.69314718055994531f : -INFINITY;
  const int pr = row0 + row;
  const int tok = pr / G;
  const bool row_ok = tok < p.S;
  const long long orow = ((long long)req * p.S + (row_ok ? tok : 0)) * p.Hq + kvh * G + pr % G;
  float acc[CPT];
#pragma unroll
  for (int c = 0; c < CPT; ++c) {
    float a = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) a += wt[w] * mb[(w * 16 + row) * (D + 2) + c0 + c];
    acc[c] = a * inv;
  }
  // Split-KV chunks (K4): publish this chunk's normalised O and log-sum-exp;
  // the last CTA to finish a chunk of a (request, KV head, row tile) merges
  // all its chunks, its own included, in a fixed order (the same arithmetic
  // whichever CTA is last):  lse = log sum_s exp(lse_s),  O = sum_s exp(lse_s - lse) O_s.
  // Every consumer thread passes the two barriers, rows past the last token too.
  volatile int* last_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 8 * (2 * L::NS + 1) + 4);
  if constexpr (kShare) {
    // this row's member: its request's partial record k of P (records of
    // request r: base[r] + k, each [Hkv][S G rows])
    const int mi = row / SG, wr = row % SG;
    const bool mine = mi < n_mem;
    const int r = mine ? mem[4 * mi] : 0;
    const long long rec0 = (long long)p.work.base[r] * p.Hkv + kvh;   // record k at rec0 + k * Hkv
    if (mine) {
      const long long at = (rec0 + (long long)mem[4 * mi + 1] * p.Hkv) * SG + wr;
      float* po = p.part_o + at * D + c0;
#pragma unroll
      for (int c = 0; c < CPT; c += 4)
        *reinterpret_cast<float4*>(po + c) = make_float4(acc[c], acc[c + 1], acc[c + 2], acc[c + 3]);
      if ((tid & 7) == 0) p.part_lse[at] = lse;
    }
    __threadfence();
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (tid < n_mem)
      mem[4 * tid + 3] = (atomicAdd(&p.unit_cnt[mem[4 * tid] * p.Hkv + kvh], 1) == mem[4 * tid + 2] - 1) ? 1 : 0;
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (!mine || mem[4 * mi + 3] == 0) return;
    __threadfence();
    const long long orow_m = ((long long)r * p.S + wr / G) * p.Hq + kvh * G + wr % G;
    merge_records<D>(p, mem[4 * mi + 2], [&](int k) { return (rec0 + (long long)k * p.Hkv) * SG + wr; }, c0,
                     orow_m, tid);
    return;
  }
  if (nsplit <= 1) {
    if (!row_ok) return;
    uint4* dst = reinterpret_cast<uint4*>(p.out + orow * D + c0);
#pragma unroll
    for (int c = 0; c < CPT; c += 8)
      dst[c / 8] = make_uint4(pack_bf16(acc[c], acc[c + 1]), pack_bf16(acc[c + 2], acc[c + 3]),
                              pack_bf16(acc[c + 4], acc[c + 5]), pack_bf16(acc[c + 6], acc[c + 7]));
    if ((tid & 7) == 0 && p.lse_out) p.lse_out[orow] = lse;
    return;
  }
  float* po = p.part_o + ((long long)cta * kMmaRows + row) * D + c0;
#pragma unroll
  for (int c = 0; c < CPT; c += 4) *reinterpret_cast<float4*>(po + c) = make_float4(acc[c], acc[c + 1], acc[c + 2], acc[c + 3]);
  if ((tid & 7) == 0) p.part_lse[(long long)cta * kMmaRows + row] = lse;
  __threadfence();
  asm volatile("bar.sync 1, 128;" ::: "memory");
  if (tid == 0) {
    const int unit = (req * p.Hkv + kvh) * p.work.row_tiles + rt;
    *last_flag = (atomicAdd(&p.unit_cnt[unit], 1) == nsplit - 1) ? 1 : 0;
  }
  asm volatile("bar.sync 1, 128;" ::: "memory");
  if (*last_flag == 0 || !row_ok) return;
  __threadfence();
  const long long c_0 = p.work.base[req] + (long long)kvh * p.work.row_tiles + rt;   // CTA of split 0
  const long long c_stride = (long long)p.Hkv * p.work.row_tiles;
  merge_records<D>(p, nsplit, [&](int sp) { return (c_0 + sp * c_stride) * kMmaRows + row; }, c0, orow, tid);
}

template <int D, bool kLayout, bool kShare>
static cudaError_t launch_attn_mma_t(const AttnParams& p, cudaStream_t st) {
  using L = MmaLayout<D, kShare>;
  cudaError_t e =
      cudaFuncSetAttribute(attn_mma_kernel<D, kLayout, kShare>, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM);
  if (e != cudaSuccess) return e;
  return launch_pdl(attn_mma_kernel<D, kLayout, kShare>, dim3(p.work.n_cta), dim3(160), (size_t)L::SMEM, st, 0, p);
}

template <int D>
static cudaError_t launch_attn_mma_d(const AttnParams& p, cudaStream_t st) {
  // shared reads are planned only where every query sees every artifact slot
  // (online spans, if any, all before the queries), so they need no layout rule
  if (p.work.share) return launch_attn_mma_t<D, false, true>(p, st);
  return p.plan.has_spans ? launch_attn_mma_t<D, true, false>(p, st) : launch_attn_mma_t<D, false, false>(p, st);
}

cudaError_t launch_attn_mma(const AttnParams& p, int D, cudaStream_t st) {
  if (D == 128) return launch_attn_mma_d<128>(p, st);
  if (D == 64) return launch_attn_mma_d<64>(p, st);
  return cudaErrorInvalidValue;
}

// APE's calibrated combination of the context and online parts (see
// ApeParams): one warp per output row (request, token, head), each lane D/32
// consecutive columns.
__global__ void __launch_bounds__(256) ape_combine_kernel(const __grid_constant__ ApeParams p, long long rows) {
  grid_dep_wait();   // the online part comes from the attention launch just before
  const long long row = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const int req = (int)(row / ((long long)p.S * p.Hq));
  const float lo = p.lse_on[row];
  const float lc = (p.t_art[req] > 0 && p.lse_ctx[row] != -INFINITY) ? p.scale * p.lse_ctx[row] : -INFINITY;
  const float m = fmaxf(lc, lo);
  const float wc = (lc == -INFINITY) ? 0.f : expf(lc - m);
  const float wo = expf(lo - m);
  const float inv = 1.f / (wc + wo);
  const int cpl = p.D / 32;   // 2 or 4
  const long long at = row * p.D + lane * cpl;
  float y[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    if (k < cpl) {
      const float c = (wc > 0.f) ? __bfloat162float(p.o_ctx[at + k]) : 0.f;
      y[k] = (wc * c + wo * __bfloat162float(p.o_on[at + k])) * inv;
    }
  }
  if (cpl == 4)
    *reinterpret_cast<uint2*>(p.out + at) = make_uint2(pack_bf16(y[0], y[1]), pack_bf16(y[2], y[3]));
  else
    *reinterpret_cast<uint32_t*>(p.out + at) = pack_bf16(y[0], y[1]);
  if (lane == 0 && p.lse_out) p.lse_out[row] = m + logf(wc + wo);
}

cudaError_t launch_ape_combine(const ApeParams& p, cudaStream_t st) {
  const long long rows = (long long)p.n_req * p.S * p.Hq;
  if (rows == 0) return cudaSuccess;
  return launch_pdl(ape_combine_kernel, dim3((unsigned)((rows * 32 + 255) / 256)), dim3(256), 0, st, 0, p, rows);
}

}  // namespace att
