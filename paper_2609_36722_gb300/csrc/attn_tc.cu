// attn_tc.cu - K2: attention of the online queries over the assembled
// artifact KV followed by the suffix KV (Sec. 2.2 Eq. routing-oracle with
// the causal mask M_t; App. A.5: SDPA with position ids of the assembled
// context), as a tcgen05 / TMEM / TMA flash-attention kernel.
//
// One CTA = 128 "packed" query rows of one request and one KV head: the G
// query heads that share the KV head are stacked into the M dimension
// (packed row = token * G + head_in_group), and one split-KV chunk of the
// request's virtual block list (artifact blocks from the block table in
// runtime order, then 64-token chunks of the suffix KV).
//
// Per 128-key tile (two 64-token blocks, each one 16 KiB TMA box pair):
//   S  = Q K^T     tcgen05.mma M=128 N=128 K=D   -> TMEM (double buffered)
//   P  = exp2(S * log2(e)/sqrt(D) - m)           softmax warps, fp32, -> bf16 smem
//   O += P V       tcgen05.mma M=128 N=D K=128   -> TMEM
// The MMA warp issues QK^T of tile j+1 before PV of tile j, so the tensor
// pipe computes while the softmax warps work on tile j.  The running max is
// only moved when it grows by more than 2^8 (then O in TMEM is rescaled), so
// most tiles need no O round trip.
//
// Warp 0: TMA producer.  Warp 1: TMEM owner and single-thread MMA issuer.
// Warps 2..5: softmax + epilogue, one query row per thread (TMEM lane).
#include <math.h>

#include "kernels.h"

namespace att {

template <int D>
struct TcLayout {
  static constexpr int NH = D / 64;                 // 64-column (128-byte) halves
  static constexpr int NS = 2;                      // K/V pipeline stages
  static constexpr int HALF = 128 * 128;            // 128 rows x 128 B
  static constexpr int Q_OFF = 0;
  static constexpr int K_OFF = Q_OFF + NH * HALF;
  static constexpr int V_OFF = K_OFF + NS * NH * HALF;
  static constexpr int P_OFF = V_OFF + NS * NH * HALF;
  static constexpr int BAR_OFF = P_OFF + 2 * HALF;
  static constexpr int LIST_OFF = BAR_OFF + 1024;
  static constexpr int SMEM = LIST_OFF + kMaxChunkBlocks * 4 + 1024;
  static constexpr uint32_t TMEM_COLS = 512;        // S0 | S1 | O
  static constexpr uint32_t S_COL0 = 0, S_COL1 = 128, O_COL = 256;
};

enum : int {
  B_Q = 0, B_KF = 1, B_VF = 3, B_KE = 5, B_VE = 7, B_SF = 9, B_SE = 11,
  B_PF = 13, B_PV = 14, B_O = 15, B_DRAIN = 16, B_NEVER = 17, B_COUNT = 18
};

// load the K (or V) half-tiles of block slot `e` into `dst` (two 64-column halves at +HALF)
template <int D>
__device__ __forceinline__ void load_slot(uint32_t dst, int e, const CUtensorMap* pool,
                                          const CUtensorMap* suf, uint32_t bar, int kvh, int Hkv,
                                          int req, int pool_rows) {
  using L = TcLayout<D>;
#pragma unroll
  for (int h = 0; h < L::NH; ++h) {
    if (e < 0) {
      const int chunk = -e - 1;
      tma_load_4d(dst + h * L::HALF, suf, bar, h * 64, kvh, chunk * kBlockTokens, req);
    } else if ((e & 127) != 0) {
      const int blk = e >> 7;
      tma_load_2d(dst + h * L::HALF, pool, bar, h * 64, (blk * Hkv + kvh) * kBlockTokens);
    } else {
      // no block: a box entirely past the end of the pool reads zeros
      tma_load_2d(dst + h * L::HALF, pool, bar, h * 64, pool_rows);
    }
  }
}

template <int D>
__global__ void __launch_bounds__(192, 1) attn_tc_kernel(const __grid_constant__ AttnParams p) {
  using L = TcLayout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR_OFF);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::BAR_OFF + 512);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 520);
  int* list = reinterpret_cast<int*>(smem + L::LIST_OFF);
  auto bar = [&](int i) { return smem_u32(&bars[i]); };

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int G = p.G;

  // ---- which (request, kv head, row tile, split) this CTA owns
  const int cta = blockIdx.x;
  const int req = find_req(p.work, cta);
  int rel = cta - p.work.base[req];
  const int rt = rel % p.work.row_tiles;
  rel /= p.work.row_tiles;
  const int kvh = rel % p.Hkv;
  const int split = rel / p.Hkv;
  const int nsplit = p.work.nsplit[req];
  const int boff = p.plan.blk_off[req];
  const int nab = p.plan.blk_off[req + 1] - boff;
  const int nsuf = (p.S_kv + kBlockTokens - 1) / kBlockTokens;
  const int row0 = rt * kTcRows;
  const int last_row = min(row0 + kTcRows - 1, p.S * G - 1);
  const int last_vis = nab + ((p.S_kv - p.S) + last_row / G) / kBlockTokens;
  const int b0 = split * p.work.chunk_blocks;
  const int b1 = min(min(b0 + p.work.chunk_blocks, nab + nsuf), last_vis + 1);
  const int nblk = max(0, b1 - b0);
  const int ntile = (nblk + 1) / 2;
  const int pool_rows = p.plan.pool_blocks * p.Hkv * kBlockTokens;

  // ---- block list of this chunk: >0 artifact (block << 7 | valid), <0 suffix chunk, 0 none
  for (int i = threadIdx.x; i < 2 * ntile; i += blockDim.x) {
    int e = 0;
    if (i < nblk) {
      const int b = b0 + i;
      if (b < nab) {
        e = p.plan.blocks[boff + b];
        const int blk = e >> 7, valid = e & 127;
        if (blk < 0 || blk >= p.plan.pool_blocks || valid < 1 || valid > kBlockTokens) {
          set_status(p.status, ATTUNER_ERR_DEVICE_CHECK);
          e = 0;
        }
      } else {
        e = -(b - nab + 1);
      }
    }
    list[i] = e;
  }
  if (threadIdx.x == 0) {
    for (int i = 0; i < B_COUNT; ++i) {
      const bool multi = (i == B_SE || i == B_SE + 1 || i == B_PF);
      mbar_init(bar(i), multi ? 4u : 1u);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), L::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ================= TMA producer =================
    if (lane == 0 && ntile > 0) {
      tma_prefetch_desc(&p.tm_q);
      tma_prefetch_desc(&p.tm_kpool);
      tma_prefetch_desc(&p.tm_vpool);
      mbar_expect_tx(bar(B_Q), L::NH * L::HALF);
#pragma unroll
      for (int h = 0; h < L::NH; ++h)
        tma_load_5d(sbase + L::Q_OFF + h * L::HALF, &p.tm_q, bar(B_Q), h * 64, 0, kvh,
                    rt * (kTcRows / G), req);
      int issued_k = 0, issued_v = 0;
      constexpr uint32_t tile_bytes = 2 * L::NH * (kBlockTokens * 128);
      for (int j = 0; j < ntile; ++j) {
        const int st = j % L::NS;
        const int e0 = list[2 * j], e1 = list[2 * j + 1];
        if (j >= L::NS &&
            !mbar_wait(bar(B_KE + st), ((j / L::NS) - 1) & 1, abort_flag, p.wait_limit, p.status))
          break;
        const uint32_t kd = sbase + L::K_OFF + st * L::NH * L::HALF;
        mbar_expect_tx(bar(B_KF + st), tile_bytes);
        load_slot<D>(kd, e0, &p.tm_kpool, &p.tm_ksuf, bar(B_KF + st), kvh, p.Hkv, req, pool_rows);
        load_slot<D>(kd + kBlockTokens * 128, e1, &p.tm_kpool, &p.tm_ksuf, bar(B_KF + st), kvh,
                     p.Hkv, req, pool_rows);
        issued_k = j + 1;
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
  } else if (warp == 1) {
    // ================= MMA issuer (one thread) =================
    if (lane == 0 && ntile > 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(128, 128, 0, 0);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, 0, 1);
      bool ok = mbar_wait(bar(B_Q), 0, abort_flag, p.wait_limit, p.status);
      bool any = false;
      auto issue_pv = [&](int i) -> bool {
        const int st = i % L::NS;
        if (!mbar_wait(bar(B_PF), i & 1, abort_flag, p.wait_limit, p.status)) return false;
        if (!mbar_wait(bar(B_VF + st), (i / L::NS) & 1, abort_flag, p.wait_limit, p.status)) return false;
        tc_fence_after();
        const uint32_t v_s = sbase + L::V_OFF + st * L::NH * L::HALF;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const uint64_t a = sdesc_sw128(sbase + L::P_OFF + (k / 4) * L::HALF + (k % 4) * 32, 16, 1024);
          const uint64_t b = sdesc_sw128(v_s + k * 2048, L::HALF, 1024);
          umma_bf16(tmem + L::O_COL, a, b, idesc_pv, (i > 0 || k > 0) ? 1u : 0u);
        }
        umma_commit(bar(B_PV));
        umma_commit(bar(B_VE + st));
        return true;
      };
      for (int j = 0; ok && j < ntile; ++j) {
        const int st = j % L::NS, sb = j & 1;
        if (!mbar_wait(bar(B_KF + st), (j / L::NS) & 1, abort_flag, p.wait_limit, p.status)) { ok = false; break; }
        if (j >= 2 && !mbar_wait(bar(B_SE + sb), ((j / 2) - 1) & 1, abort_flag, p.wait_limit, p.status)) { ok = false; break; }
        tc_fence_after();
        const uint32_t k_s = sbase + L::K_OFF + st * L::NH * L::HALF;
#pragma unroll
        for (int k = 0; k < D / 16; ++k) {
          const uint32_t off = (k / 4) * L::HALF + (k % 4) * 32;
          umma_bf16(tmem + (sb ? L::S_COL1 : L::S_COL0), sdesc_sw128(sbase + L::Q_OFF + off, 16, 1024),
                    sdesc_sw128(k_s + off, 16, 1024), idesc_qk, k > 0 ? 1u : 0u);
        }
        any = true;
        umma_commit(bar(B_SF + sb));
        umma_commit(bar(B_KE + st));
        if (j >= 1 && !issue_pv(j - 1)) { ok = false; break; }
      }
      if (ok) ok = issue_pv(ntile - 1);
      if (ok) {
        umma_commit(bar(B_O));
      } else if (any) {
        umma_commit(bar(B_DRAIN));
        mbar_drain(bar(B_DRAIN), 0, p.status);
      }
    }
  } else {
    // ================= softmax + epilogue (warps 2..5) =================
    const int q = warp & 3;
    const int r = q * 32 + lane;                 // tile row == TMEM lane
    const int pr = row0 + r;                     // packed row
    const int tok = pr / G, jh = pr % G;
    const int lim = (p.S_kv - p.S) + tok;        // last visible suffix key
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    if (p.inject_stuck && q == 2)
      ok = warp_wait(bar(B_NEVER), 0, abort_flag, p.wait_limit, p.status);   // nothing arrives: times out
    for (int j = 0; ok && j < ntile; ++j) {
      const int sb = j & 1;
      if (!warp_wait(bar(B_SF + sb), (j / 2) & 1, abort_flag, p.wait_limit, p.status)) { ok = false; break; }
      tc_fence_after();
      float s[128];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_base + (sb ? L::S_COL1 : L::S_COL0) + c * 32, s + c * 32);
      tc_wait_ld();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(B_SE + sb));

      // mask: artifact block tails, suffix causality, empty slots
#pragma unroll
      for (int b = 0; b < 2; ++b) {
        const int e = list[2 * j + b];
        if (e > 0) {
          const int valid = e & 127;
          if (valid < kBlockTokens) {
#pragma unroll
            for (int c = 0; c < 64; ++c) if (c >= valid) s[64 * b + c] = -INFINITY;
          }
        } else if (e < 0) {
          const int kbase = (-e - 1) * kBlockTokens;
          if (kbase + kBlockTokens - 1 > lim) {
#pragma unroll
            for (int c = 0; c < 64; ++c) if (kbase + c > lim) s[64 * b + c] = -INFINITY;
          }
        } else {
#pragma unroll
          for (int c = 0; c < 64; ++c) s[64 * b + c] = -INFINITY;
        }
      }
      // row max: eight independent chains of 3-input max, then a small tree
      float mk[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) mk[k] = fmaxf(s[k], s[k + 8]);
#pragma unroll
      for (int c = 16; c < 128; c += 16) {
#pragma unroll
        for (int k = 0; k < 8; ++k) mk[k] = fmax3(mk[k], s[c + k], s[c + k + 8]);
      }
      float mx = fmax3(fmax3(mk[0], mk[1], mk[2]), fmax3(mk[3], mk[4], mk[5]), fmaxf(mk[6], mk[7]));
      mx *= p.scale_log2;
      float alpha = 1.f;
      if (mx > m_run + 8.f) {              // move the reference max only when it grows past 2^8
        alpha = ex2(m_run - mx);           // m_run = -inf gives 0
        m_run = mx;
      }
      const float neg = (m_run == -INFINITY) ? 0.f : -m_run;
      // p = 2^(s * log2(e)/sqrt(d) - m): packed fp32 FMA, then ex2; row sum in 8 packed chains
      const uint64_t sc2 = f2_pack(p.scale_log2, p.scale_log2), ng2 = f2_pack(neg, neg);
      uint64_t acc2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
      for (int c = 0; c < 128; c += 2) {
        float a, b;
        f2_unpack(f2_fma(f2_pack(s[c], s[c + 1]), sc2, ng2), a, b);
        s[c] = ex2(a);
        s[c + 1] = ex2(b);
        acc2[(c >> 1) & 3] = f2_add(acc2[(c >> 1) & 3], f2_pack(s[c], s[c + 1]));
      }
      float rs;
      {
        float a0, a1;
        f2_unpack(f2_add(f2_add(acc2[0], acc2[1]), f2_add(acc2[2], acc2[3])), a0, a1);
        rs = a0 + a1;
      }
      l_run = l_run * alpha + rs;

      // PV of the previous tile must be done: P buffer free, O current
      if (j >= 1 && !warp_wait(bar(B_PV), (j - 1) & 1, abort_flag, p.wait_limit, p.status)) { ok = false; break; }
#pragma unroll
      for (int h = 0; h < 2; ++h) {
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const float* f = s + 64 * h + 8 * c;
          st_shared_v4(sbase + L::P_OFF + h * L::HALF + sw128_off(r, c), pack_bf16(f[0], f[1]),
                       pack_bf16(f[2], f[3]), pack_bf16(f[4], f[5]), pack_bf16(f[6], f[7]));
        }
      }
      if (j >= 1 && __any_sync(0xffffffffu, alpha != 1.f)) {
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          float o[32];
          tmem_ld32(tmem + lane_base + L::O_COL + c * 32, o);
          tc_wait_ld();
#pragma unroll
          for (int k = 0; k < 32; ++k) o[k] *= alpha;
          tmem_st32(tmem + lane_base + L::O_COL + c * 32, o);
        }
        tc_wait_st();
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(B_PF));
    }

    // ---- epilogue
    const bool split_out = nsplit > 1;
    if (ok && ntile > 0) ok = warp_wait(bar(B_O), 0, abort_flag, p.wait_limit, p.status);
    if (ok) {
      tc_fence_after();
      const float inv_l = (l_run > 0.f) ? 1.f / l_run : 0.f;
      const float lse = (l_run > 0.f) ? (m_run + log2f(l_run)) * 0.69314718055994531f : -INFINITY;
      const bool row_ok = tok < p.S;
      if (split_out) {
        float* po = p.part_o + ((long long)cta * kTcRows + r) * D;
        if (ntile > 0) {
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            float o[32];
            tmem_ld32(tmem + lane_base + L::O_COL + c * 32, o);
            tc_wait_ld();
            if (row_ok) {
#pragma unroll
              for (int k = 0; k < 32; k += 4)
                *reinterpret_cast<float4*>(po + c * 32 + k) =
                    make_float4(o[k] * inv_l, o[k + 1] * inv_l, o[k + 2] * inv_l, o[k + 3] * inv_l);
            }
          }
        }
        if (row_ok) p.part_lse[(long long)cta * kTcRows + r] = lse;
      } else if (ntile > 0) {
        const long long orow = ((long long)req * p.S + tok) * p.Hq + kvh * G + jh;
        uint4* dst = reinterpret_cast<uint4*>(p.out + orow * D);
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          float o[32];
          tmem_ld32(tmem + lane_base + L::O_COL + c * 32, o);
          tc_wait_ld();
          if (row_ok) {
#pragma unroll
            for (int k = 0; k < 4; ++k)
              dst[c * 4 + k] = make_uint4(
                  pack_bf16(o[8 * k] * inv_l, o[8 * k + 1] * inv_l), pack_bf16(o[8 * k + 2] * inv_l, o[8 * k + 3] * inv_l),
                  pack_bf16(o[8 * k + 4] * inv_l, o[8 * k + 5] * inv_l), pack_bf16(o[8 * k + 6] * inv_l, o[8 * k + 7] * inv_l));
          }
        }
        if (row_ok && p.lse_out) p.lse_out[orow] = lse;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, L::TMEM_COLS);
  }
}

template <int D>
static cudaError_t launch_attn_tc_t(const AttnParams& p, cudaStream_t st) {
  using L = TcLayout<D>;
  cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM);
  if (e != cudaSuccess) return e;
  attn_tc_kernel<D><<<p.work.n_cta, 192, L::SMEM, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_attn_tc(const AttnParams& p, int D, cudaStream_t st) {
  if (D == 128) return launch_attn_tc_t<128>(p, st);
  if (D == 64) return launch_attn_tc_t<64>(p, st);
  return cudaErrorInvalidValue;
}

}  // namespace att
