// qproj.cuh - K1b: the adapted query projection of Sec. 3, Eq.
// (query-adaptation), followed by the model's original query RMSNorm and
// RoPE, as one tcgen05 GEMM with a fused epilogue:
//
//   Q[m, h, :] = RoPE( RMSNorm( x_m W_q,h^T + bf16(s * x_m A^T) B_h^T ) * w, pos_m )
//
// A CTA computes MR x 128 query rows (MR = 1 or 2 TMEM accumulators) of one
// whole head, so the RMSNorm and every RoPE pair (j, j + D/2) stay inside one
// CTA.  Each 64-wide K block stages the MR x tiles, the head's W_q rows and,
// right below them, the r rows of the LoRA A matrix, so ONE MMA of N = D + r
// per accumulator produces both x W_q,h^T (columns 0..D-1) and u = x A^T
// (columns D..D+r-1).
//
// The K dimension is split over a thread-block cluster of KS = 1, 2, 4 or 8
// CTAs (cluster rank = K slice).  At the sizes of a prefill suffix or a decode
// step the operand bytes that reach each SM bound this kernel, not the tensor
// core: a CTA receives (MR*128 + D + r) * hidden/KS * 2 bytes, so two
// accumulators sharing each W tile and K slices shared by a cluster cut both
// the x tile every head re-reads and each SM's share of W_q.  After the K loop
// every CTA writes the fp32 partial rows that each peer owns (CTA k owns rows
// [k, k+1) * MR*128/KS of the tile) into that peer's shared memory (the idle
// stage ring) with distributed shared-memory stores.  After a cluster barrier
// each CTA sums its rows' KS partials in slice order (so the result does not
// depend on which CTA finished first), adds the rank-r update
// bf16(s * u) B_h^T, and finishes the RMSNorm, RoPE and bf16 store with
// KS/MR threads per row.  The rank-r update is one more MMA on the
// tensor core: bf16(s * u) is written as a small K-major tile in shared
// memory and multiplied by B_h^T (with KS = 1 it accumulates straight into the
// accumulator; with KS > 1, after the exchange, into freed TMEM columns that
// each thread adds to its own).
//
// Warp 0: TMA producer; warp 1: TMEM owner + MMA issuer; warps 2..5:
// epilogue (TMEM lane quadrants 2, 3, 0, 1; tcgen05.ld 32x32b).
#pragma once

#include "kernels.h"

namespace att {

template <int D, int MR>
struct QpLayout {
  static constexpr int X_BYTES = 128 * 128;               // one x tile: 128 rows x 64 bf16 (SW128)
  static constexpr int W_OFF = MR * X_BYTES;               // the head's D rows of W_q x 64 bf16 ...
  static constexpr int A_OFF = W_OFF + D * 128;            // ... then up to 64 rows of LoRA A
  static constexpr int STAGE = qp_stage_bytes(D, MR);
  static constexpr int NS = (200 * 1024) / STAGE;          // 5/3 stages (D = 128), 6/4 (D = 64)
  static constexpr int RING = qp_ring_bytes(D, MR);
  static_assert(STAGE == A_OFF + 64 * 128 && RING == NS * STAGE, "stage layout");
  static constexpr int B_OFF = RING;                       // B_h: [r/8][D rows][8 bf16], no swizzle
  static constexpr int BAR_OFF = B_OFF + 64 * D * 2;
  static constexpr int SMEM = BAR_OFF + 256 + 1024;       // + alignment slack
  static constexpr uint32_t TMEM_COLS = MR == 2 ? 512 : 256;
  static constexpr uint32_t ACC_STRIDE = 256;              // accumulator a at TMEM column 256 a
};

// Shared-memory matrix descriptor, no swizzle (canonical K-major layout of
// 8-row x 16-byte core matrices): lbo = byte distance between the two
// 8-element K halves of a core-matrix pair, sbo = between 8-row groups.
ATT_DEV uint64_t sdesc_noswz(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  return d;
}

ATT_DEV void st_cluster_v4(uint32_t caddr, float a, float b, float c, float d) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(caddr), "f"(a), "f"(b), "f"(c),
               "f"(d)
               : "memory");
}

enum : int { QB_ACC = 0, QB_LORA = 1, QB_LUP = 2, QB_DRAIN = 3, QB_FULL = 4 };   // + NS full, NS empty

// RMSNorm * w, RoPE and the bf16 store of one row's columns held by this
// thread: v[0, NP) are columns jlo + [0, NP), v[NP, 2 NP) columns
// D/2 + jlo + [0, NP).  The TPR consecutive lanes that share a row add their
// sums of squares with a butterfly (every lane gets the same sum).  Rows past
// M store nothing; V heads (K/V mode) are stored as projected.
template <int D, int NP, int TPR>
ATT_DEV void qproj_finish(const QprojParams& p, float* v, int m, int head, bool is_v, int jlo, bool store) {
  const bool row_ok = m < p.M;
  const int mr = row_ok ? m : p.M - 1;
  if (!is_v) {
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < 2 * NP; ++j) ss = fmaf(v[j], v[j], ss);
#pragma unroll
    for (int o = 1; o < TPR; o <<= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    const float rinv = rsqrtf(ss * (1.0f / D) + p.eps);
#pragma unroll
    for (int c = 0; c < NP; ++c) {
      const int j = jlo + c;
      const float2 cs = p.rope[(long long)j * p.M + mr];
      const float a = v[c] * rinv * __bfloat162float(p.qnorm_w[j]);
      const float b = v[c + NP] * rinv * __bfloat162float(p.qnorm_w[j + D / 2]);
      v[c] = a * cs.x - b * cs.y;
      v[c + NP] = b * cs.x + a * cs.y;
    }
  }
  if (store && row_ok) {
    const long long t = (long long)(m / p.S) * p.S_out + (p.S_out - p.S) + m % p.S;   // output token row
    __nv_bfloat16* base = is_v ? p.out2 : p.q_out;
    __nv_bfloat16* orow = base + (t * p.Hout + head) * D;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      uint4* dst = reinterpret_cast<uint4*>(orow + h * (D / 2) + jlo);
      const float* src = v + h * NP;
#pragma unroll
      for (int c = 0; c < NP / 8; ++c)
        dst[c] = make_uint4(pack_bf16(src[8 * c], src[8 * c + 1]), pack_bf16(src[8 * c + 2], src[8 * c + 3]),
                            pack_bf16(src[8 * c + 4], src[8 * c + 5]), pack_bf16(src[8 * c + 6], src[8 * c + 7]));
    }
  }
}

// Epilogue without a K split: one accumulator row per thread and
// accumulator; the rank-r update runs on the tensor core.  R = LoRA rank
// rounded up to 16 (0: no adapter).  `ok` is uniform over the 128 threads.
template <int D, int MR, int R>
ATT_DEV void qproj_epilogue_direct(const QprojParams& p, uint8_t* smem, uint32_t tmem, uint64_t* bars,
                                   volatile int* abort_flag, int head, bool is_v, int m0, bool ok) {
  using L = QpLayout<D, MR>;
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int q = warp & 3;
  const int r = q * 32 + lane;                   // accumulator row (TMEM lane) of this thread
  const uint32_t lane_t = (uint32_t)(q * 32) << 16;
  auto bar = [&](int i) { return smem_u32(&bars[i]); };

  if constexpr (R > 0) if (ok) {
    // U_a = bf16(s * u) of accumulator a as a K-major tile [R/8][128 rows][8] in
    // the idle stage ring, then per 16 of R one MMA: acc_a[:, 0..D) += U_a B_h^T
#pragma unroll
    for (int a = 0; a < MR; ++a) {
      float u[32 * ((R + 31) / 32)];
#pragma unroll
      for (int c = 0; c < (R + 31) / 32; ++c) tmem_ld32(tmem + lane_t + a * L::ACC_STRIDE + D + c * 32, u + c * 32);
      tc_wait_ld();
#pragma unroll
      for (int g = 0; g < R / 8; ++g) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int k = g * 8 + 2 * e;
          w[e] = pack_bf16(k < p.r ? p.s * u[k] : 0.f, k + 1 < p.r ? p.s * u[k + 1] : 0.f);
        }
        st_shared_v4(sbase + (a * (R / 8) + g) * 2048 + r * 16, w[0], w[1], w[2], w[3]);
      }
    }
    fence_proxy_async_smem();
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (threadIdx.x == 64) {
      if (mbar_wait(bar(QB_LORA), 0, abort_flag, p.wait_limit, p.status)) {
        tc_fence_after();
        constexpr uint32_t idesc = idesc_bf16_f32(128, D, 0, 0);
#pragma unroll
        for (int a = 0; a < MR; ++a)
#pragma unroll
          for (int kk = 0; kk < R / 16; ++kk)
            umma_bf16(tmem + a * L::ACC_STRIDE, sdesc_noswz(sbase + (a * (R / 8) + 2 * kk) * 2048, 2048, 128),
                      sdesc_noswz(sbase + L::B_OFF + kk * 2 * (D * 16), D * 16, 128), idesc, 1u);
        umma_commit(bar(QB_LUP));
      } else {
        mbar_arrive(bar(QB_LUP));       // never issued: release the waiters (status already TIMEOUT)
      }
    }
    warp_wait(bar(QB_LUP), 0, abort_flag, p.wait_limit, p.status);
    tc_fence_after();
  }
#pragma unroll 1
  for (int a = 0; a < MR; ++a) {
    float v[D];
    if (ok) {
#pragma unroll
      for (int c = 0; c < D / 32; ++c) tmem_ld32(tmem + lane_t + a * L::ACC_STRIDE + c * 32, v + c * 32);
      tc_wait_ld();
    }
    qproj_finish<D, D / 2, 1>(p, v, m0 + a * 128 + r, head, is_v, 0, ok);
  }
}

// Value k of this thread's NP columns inside a 32-column chunk `t` that
// starts `off` columns before them (off a multiple of NP below 32, the same
// for no two threads of a row): a select chain, so `t` stays in registers.
template <int NP>
ATT_DEV float chunk_pick(const float* t, int off, int k) {
  float x = t[k];
#pragma unroll
  for (int o = NP; o < 32; o += NP) x = (off == o) ? t[o + k] : x;
  return x;
}

// Epilogue of a K slice `ks` of a cluster of KS: exchange of the partial rows,
// the fixed-order sum over the slices, the rank-r update and the finish with
// TPR = KS/MR threads per row.  Called by the 128 epilogue threads after the
// first cluster barrier (every peer's MMAs are complete and its stage ring is
// free); contains the second one.  The rank-r update runs on the tensor core:
// each thread writes bf16(s * u) of its row into row (its TMEM lane) of a
// K-major tile (the TPR threads of a row write TPR copies), one MMA per 16 of
// R puts U B_h^T into the freed columns of accumulator 0, and every thread
// adds its own columns from its own lane.
template <int D, int MR, int KS, int R>
ATT_DEV void qproj_epilogue_split(const QprojParams& p, uint8_t* smem, uint32_t tmem, uint64_t* bars,
                                  volatile int* abort_flag, int head, bool is_v, int m0, int ks, bool ok) {
  using L = QpLayout<D, MR>;
  constexpr int W = D + R;                       // partial columns: x W^T, then u = x A^T
  constexpr int WP = qp_pitch(W);
  constexpr int ROWS = MR * 128 / KS;            // rows owned by each CTA of the cluster
  constexpr int TPR = KS / MR;                   // threads per owned row
  constexpr int NP = D / 2 / TPR;                // rotary pairs per thread
  static_assert(TPR >= 1 && NP >= 8 && qp_recv_bytes(MR, D, R) <= L::RING, "unsupported split shape");
  const uint32_t sbase = smem_u32(smem);         // exchange buffer [KS slices][ROWS][WP] fp32 over the ring
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int q = warp & 3;
  const int et = threadIdx.x - 64;
  const uint32_t lane_t = (uint32_t)(q * 32) << 16;
  auto bar = [&](int i) { return smem_u32(&bars[i]); };

  if (ok) {
#pragma unroll 1
    for (int a = 0; a < MR; ++a) {
      const int row = a * 128 + q * 32 + lane;
      const bool valid = m0 + row < p.M;
      const uint32_t dst = dsmem_addr(sbase + (uint32_t)((ks * ROWS + row % ROWS) * WP) * 4u, row / ROWS);
#pragma unroll
      for (int c = 0; c < (W + 31) / 32; ++c) {
        float t[32];
        tmem_ld32(tmem + lane_t + a * L::ACC_STRIDE + c * 32, t);
        tc_wait_ld();
        if (valid) {
#pragma unroll
          for (int k = 0; k < 32; k += 4)
            if (c * 32 + k < W) st_cluster_v4(dst + (uint32_t)(c * 32 + k) * 4u, t[k], t[k + 1], t[k + 2], t[k + 3]);
        }
      }
    }
  }
  tc_fence_before();
  cluster_sync_all();   // 2: every partial row is in its owner's shared memory

  const int lr = et / TPR, sub = et % TPR;
  const int jlo = sub * NP;
  const int m = m0 + ks * ROWS + lr;
  float v[2 * NP];
  float u[R > 0 ? R : 1];
#pragma unroll
  for (int c = 0; c < 2 * NP; ++c) v[c] = 0.f;
#pragma unroll
  for (int c = 0; c < R; ++c) u[c] = 0.f;
  const float* base = reinterpret_cast<const float*>(smem) + lr * WP;
#pragma unroll 1
  for (int k = 0; k < KS; ++k) {
    const float* src = base + k * ROWS * WP;
#pragma unroll
    for (int c = 0; c < NP; c += 4) {
      const float4 x0 = *reinterpret_cast<const float4*>(src + jlo + c);
      const float4 x1 = *reinterpret_cast<const float4*>(src + D / 2 + jlo + c);
      v[c] += x0.x; v[c + 1] += x0.y; v[c + 2] += x0.z; v[c + 3] += x0.w;
      v[NP + c] += x1.x; v[NP + c + 1] += x1.y; v[NP + c + 2] += x1.z; v[NP + c + 3] += x1.w;
    }
#pragma unroll
    for (int c = 0; c < R; c += 4) {
      const float4 x = *reinterpret_cast<const float4*>(src + D + c);
      u[c] += x.x; u[c + 1] += x.y; u[c + 2] += x.z; u[c + 3] += x.w;
    }
  }
  if constexpr (R > 0) if (ok) {
    asm volatile("bar.sync 1, 128;" ::: "memory");   // every thread is done with the exchange buffer
#pragma unroll
    for (int g = 0; g < R / 8; ++g) {
      uint32_t w[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int k = g * 8 + 2 * e;
        w[e] = pack_bf16(k < p.r ? p.s * u[k] : 0.f, k + 1 < p.r ? p.s * u[k + 1] : 0.f);
      }
      st_shared_v4(sbase + g * 2048 + (q * 32 + lane) * 16, w[0], w[1], w[2], w[3]);
    }
    fence_proxy_async_smem();
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (threadIdx.x == 64) {
      if (mbar_wait(bar(QB_LORA), 0, abort_flag, p.wait_limit, p.status)) {
        tc_fence_after();
        constexpr uint32_t idesc = idesc_bf16_f32(128, D, 0, 0);
#pragma unroll
        for (int kk = 0; kk < R / 16; ++kk)
          umma_bf16(tmem, sdesc_noswz(sbase + 2 * kk * 2048, 2048, 128),
                    sdesc_noswz(sbase + L::B_OFF + kk * 2 * (D * 16), D * 16, 128), idesc, kk > 0 ? 1u : 0u);
        umma_commit(bar(QB_LUP));
      } else {
        mbar_arrive(bar(QB_LUP));       // never issued: release the waiters (status already TIMEOUT)
      }
    }
    warp_wait(bar(QB_LUP), 0, abort_flag, p.wait_limit, p.status);
    tc_fence_after();
    // columns [32c, 32c + 32) of the update: half h, starting cb columns into it
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
      float t[32];
      tmem_ld32(tmem + lane_t + c * 32, t);
      tc_wait_ld();
      constexpr int HALF = D / 2;
      const int h = (c * 32) / HALF, cb = c * 32 - h * HALF;
      if constexpr (NP >= 32) {
        if (TPR == 1 || jlo == cb) {
#pragma unroll
          for (int k = 0; k < 32; ++k) v[h * NP + (TPR == 1 ? cb : 0) + k] += t[k];
        }
      } else {
        const int off = jlo - cb;
        if (off >= 0 && off < 32) {
#pragma unroll
          for (int k = 0; k < NP; ++k) v[h * NP + k] += chunk_pick<NP>(t, off, k);
        }
      }
    }
  }
  qproj_finish<D, NP, TPR>(p, v, m, head, is_v, jlo, ok);
}

template <int D, int MR, int KS>
__global__ void __launch_bounds__(192, 1) qproj_kernel(const __grid_constant__ QprojParams p) {
  using L = QpLayout<D, MR>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR_OFF);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::BAR_OFF + 192);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 200);
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  const int B_FULL = QB_FULL, B_EMPTY = QB_FULL + L::NS;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  // blockIdx.x = head * KS + ks (a cluster of KS along x: rank = ks)
  const int head = blockIdx.x / KS;
  const int ks = blockIdx.x % KS;
  const int m0 = blockIdx.y * (MR * 128);
  const bool is_v = p.kv && head >= p.Hout;              // K/V mode: this CTA projects V
  const int oh = is_v ? head - p.Hout : head;             // head within its output
  const CUtensorMap* tm_w = is_v ? &p.tm_w2 : &p.tm_w;
  const int n0 = oh * D;
  const int nk = p.hidden / 64;
  const int kb0 = ks * nk / KS, kb1 = (ks + 1) * nk / KS;
  const bool lora = p.n_lora > 0;
  const int nmma = D + (lora ? p.n_lora : 0);             // N of the main MMA
  const uint32_t stage_tx = MR * L::X_BYTES + D * 128 + (lora ? p.n_lora * 128 : 0);

  if (threadIdx.x == 0) {
    for (int i = 0; i < QB_FULL + 2 * L::NS; ++i) mbar_init(bar(i), 1);
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
    if (lane == 0) {
      tma_prefetch_desc(&p.tm_x);
      tma_prefetch_desc(tm_w);
      if (lora) {
        // B_h: r/8 boxes of [D rows][8 columns] (columns past r read as zeros)
        mbar_expect_tx(bar(QB_LORA), (p.n_lora / 8) * D * 16);
        for (int g = 0; g < p.n_lora / 8; ++g)
          tma_load_2d(sbase + L::B_OFF + g * D * 16, &p.tm_b, bar(QB_LORA), g * 8, n0);
      }
      int issued = 0;
      for (int kb = kb0; kb < kb1; ++kb) {
        const int it = kb - kb0, st = it % L::NS;
        if (it >= L::NS &&
            !mbar_wait(bar(B_EMPTY + st), ((it / L::NS) - 1) & 1, abort_flag, p.wait_limit, p.status))
          break;
        const uint32_t s0 = sbase + st * L::STAGE;
        mbar_expect_tx(bar(B_FULL + st), stage_tx);
#pragma unroll
        for (int a = 0; a < MR; ++a) tma_load_2d(s0 + a * L::X_BYTES, &p.tm_x, bar(B_FULL + st), kb * 64, m0 + a * 128);
        tma_load_2d(s0 + L::W_OFF, tm_w, bar(B_FULL + st), kb * 64, n0);
        if (lora) tma_load_2d(s0 + L::A_OFF, &p.tm_a, bar(B_FULL + st), kb * 64, 0);
        issued = it + 1;
      }
      if (*abort_flag) {   // let every copy this CTA issued land before exiting
        if (lora) mbar_drain(bar(QB_LORA), 0, p.status);
        for (int it = (issued > L::NS ? issued - L::NS : 0); it < issued; ++it)
          mbar_drain(bar(B_FULL + it % L::NS), (it / L::NS) & 1, p.status);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, nmma, 0, 0);
      bool ok = true;
      bool any = false;
      for (int kb = kb0; kb < kb1; ++kb) {
        const int it = kb - kb0, st = it % L::NS;
        if (!mbar_wait(bar(B_FULL + st), (it / L::NS) & 1, abort_flag, p.wait_limit, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t s0 = sbase + st * L::STAGE;
#pragma unroll
        for (int k = 0; k < 4; ++k)
#pragma unroll
          for (int a = 0; a < MR; ++a)
            umma_bf16(tmem + a * L::ACC_STRIDE, sdesc_sw128(s0 + a * L::X_BYTES + k * 32, 16, 1024),
                      sdesc_sw128(s0 + L::W_OFF + k * 32, 16, 1024), idesc, (it > 0 || k > 0) ? 1u : 0u);
        any = true;
        umma_commit(bar(B_EMPTY + st));
      }
      if (ok) {
        umma_commit(bar(QB_ACC));
      } else if (any) {
        umma_commit(bar(QB_DRAIN));
        mbar_drain(bar(QB_DRAIN), 0, p.status);
      }
    }
  } else {
    // epilogue: warps 2..5 -> TMEM lane quadrants 2, 3, 0, 1.  The RoPE table
    // comes from the prep kernel just before this one.
    grid_dep_wait();
    const bool acc_ok = warp_wait(bar(QB_ACC), 0, abort_flag, p.wait_limit, p.status);
    // one answer for all four warps: a warp that gave up raised the abort flag
    asm volatile("bar.sync 1, 128;" ::: "memory");
    const bool ok = acc_ok && *abort_flag == 0;
    if (ok) tc_fence_after();
    const int nl = lora ? p.n_lora : 0;
    if constexpr (KS == 1) {
      if (nl == 0)
        qproj_epilogue_direct<D, MR, 0>(p, smem, tmem, bars, abort_flag, oh, is_v, m0, ok);
      else if (nl <= 16)
        qproj_epilogue_direct<D, MR, 16>(p, smem, tmem, bars, abort_flag, oh, is_v, m0, ok);
      else if (nl <= 32)
        qproj_epilogue_direct<D, MR, 32>(p, smem, tmem, bars, abort_flag, oh, is_v, m0, ok);
      else
        qproj_epilogue_direct<D, MR, 64>(p, smem, tmem, bars, abort_flag, oh, is_v, m0, ok);
    } else {
      cluster_sync_all();   // 1: every CTA of the cluster is past its K loop
      if (nl == 0)
        qproj_epilogue_split<D, MR, KS, 0>(p, smem, tmem, bars, abort_flag, oh, is_v, m0, ks, ok);
      else if (nl <= 16)
        qproj_epilogue_split<D, MR, KS, 16>(p, smem, tmem, bars, abort_flag, oh, is_v, m0, ks, ok);
      else if constexpr (qp_recv_bytes(MR, D, 32) <= L::RING) {
        if (nl <= 32)
          qproj_epilogue_split<D, MR, KS, 32>(p, smem, tmem, bars, abort_flag, oh, is_v, m0, ks, ok);
        else if constexpr (qp_recv_bytes(MR, D, 64) <= L::RING)
          qproj_epilogue_split<D, MR, KS, 64>(p, smem, tmem, bars, abort_flag, oh, is_v, m0, ks, ok);
        else
          cluster_sync_all();   // (refused on the host) keep the peers' barrier count
      } else {
        cluster_sync_all();
      }
    }
  }
  if (KS > 1 && warp < 2) {
    // the epilogue's two cluster barriers count every thread of the cluster
    cluster_sync_all();
    cluster_sync_all();
  }
  // let the attention kernel launch once every CTA is here (triggering at the
  // start measured slower: its early CTAs crowd the SMs the tail needs)
  grid_dep_launch();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, L::TMEM_COLS);
  }
}

template <int D, int MR, int KS>
static cudaError_t launch_qproj_t(const QprojParams& p, cudaStream_t st) {
  using L = QpLayout<D, MR>;
  cudaError_t e = cudaFuncSetAttribute(qproj_kernel<D, MR, KS>, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM);
  if (e != cudaSuccess) return e;
  dim3 grid(p.Hq * KS, (p.M + MR * 128 - 1) / (MR * 128));
  return launch_pdl(qproj_kernel<D, MR, KS>, grid, dim3(192), (size_t)L::SMEM, st, KS > 1 ? KS : 0, p);
}

// Launch with MR accumulators and a cluster of ks K slices (each (D, MR) pair
// is instantiated in its own translation unit so that they compile in parallel).
template <int D, int MR>
cudaError_t launch_qproj_mr(const QprojParams& p, int ks, cudaStream_t st) {
  switch (ks) {
    case 1: return launch_qproj_t<D, MR, 1>(p, st);
    case 2: return launch_qproj_t<D, MR, 2>(p, st);
    case 4: return launch_qproj_t<D, MR, 4>(p, st);
    case 8:
      if constexpr (D / 2 / (8 / MR) >= 8) return launch_qproj_t<D, MR, 8>(p, st);
      return cudaErrorInvalidValue;
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace att
