// qproj.cu - K1b: the adapted query projection of Sec. 3, Eq.
// (query-adaptation), followed by the model's original query RMSNorm and
// RoPE, as one tcgen05 GEMM with a fused epilogue:
//
//   Q[m, h, :] = RoPE( RMSNorm( x_m W_q,h^T + bf16(s * x_m A^T) B_h^T ) * w, pos_m )
//
// CTA tile: 128 query rows x one head (N = D = 64 or 128), so every
// accumulator row holds a whole head and the RMSNorm needs no cross-CTA
// reduction of its own.  Each K block loads the x tile, the W_q rows of the
// head and, right below them, the r rows of the LoRA A matrix, so ONE MMA of
// N = D + r produces both x W_q,h^T (columns 0..D-1) and u = x A^T (columns
// D..D+r-1).  After the K loop the epilogue writes bf16(s * u) as a small
// K-major tile in shared memory and one MMA with B_h (loaded by TMA at the
// start) adds the rank-r update into a second TMEM accumulator.
//
// When (row tiles x heads) cannot fill half the GPU (decode, short suffixes),
// each head's columns are split over a cluster of P = 2 or 4 CTAs: CTA `part`
// computes columns j0 + [0, D/2P) and D/2 + j0 + [0, D/2P), j0 = part D/2P,
// so the RoPE pairs (j, j + D/2) stay inside one CTA, and the RMSNorm's sum of
// squares is the sum of the P partial sums, exchanged through distributed
// shared memory (summed in part order, so every part gets the same value).
// More CTAs stream W_q at once: at these sizes the operand loads, not the
// tensor core, bound the kernel.
//
// Alternatively (an option, off by default) the K dimension is split over up
// to 4 CTAs per tile; each publishes its fp32
// partial accumulators and the last CTA to arrive (an atomic counter per
// tile, cleared by the prep kernel of the same call) sums all of them in
// split order (the result does not depend on arrival order) and finishes.
//
// Warp 0: TMA producer; warp 1: TMEM owner + MMA issuer; warps 2..5:
// epilogue (one accumulator row per thread, tcgen05.ld 32x32b).
#include "kernels.h"

namespace att {

template <int D>
struct QpLayout {
  static constexpr int X_BYTES = 128 * 128;   // x tile: 128 rows x 64 bf16
  static constexpr int W_BYTES = D * 128;     // W_q rows of the head, then...
  static constexpr int A_BYTES = 64 * 128;    // ...up to 64 rows of the LoRA A matrix
  static constexpr int STAGE = X_BYTES + W_BYTES + A_BYTES;
  static constexpr int NS = (D == 128) ? 5 : 6;
  static constexpr int B_OFF = NS * STAGE;               // B_h: [r/8][D rows][8 bf16]
  static constexpr int B_BYTES = 64 * D * 2;
  static constexpr int BAR_OFF = B_OFF + B_BYTES;
  static constexpr int RED_OFF = BAR_OFF + 512;          // column split: 128 partial sums of squares
  static constexpr int SMEM = RED_OFF + 512 + 1024;     // + alignment slack
  static constexpr uint32_t TMEM_COLS = 512;            // [x W^T | x A^T] at 0, LoRA update at 256
  static constexpr uint32_t LUP_COL = 256;
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

enum : int { QB_ACC = 0, QB_LORA = 1, QB_LUP = 2, QB_DRAIN = 3, QB_FULL = 4 };   // + NS full, NS empty

// Epilogue of one accumulator row per thread (warps 2..5).  R = LoRA rank
// rounded up to 16 (0: no adapter); P = CTAs per head (column split).  `ok`
// is uniform over the 128 epilogue threads; with P > 1 every thread passes
// the two cluster barriers whatever `ok` is, so the peers never wait for it.
template <int D, int P, int R>
__device__ __forceinline__ void qproj_epilogue(const QprojParams& p, uint8_t* smem, uint32_t tmem,
                                               uint64_t* bars, volatile int* abort_flag,
                                               volatile int* last_flag, int head, int part, bool is_v,
                                               int ks, int tile, int m0, bool ok) {
  using L = QpLayout<D>;
  constexpr int DC = D / P;            // columns of this CTA: two halves of DC/2
  constexpr int RU = R > 0 ? R : 1;
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int q = warp & 3;
  const int r = q * 32 + lane;
  const int et = threadIdx.x - 64;     // 0..127 within the epilogue warps
  const int m = m0 + r;
  const int j0 = part * (DC / 2);      // first rotary pair of this CTA
  const uint32_t row_t = tmem + ((uint32_t)(q * 32) << 16);
  constexpr int rowlen = DC + R;
  auto bar = [&](int i) { return smem_u32(&bars[i]); };

  float v[DC];
  float u[RU];
  if (ok) {
#pragma unroll
    for (int c = 0; c < DC / 32; ++c) tmem_ld32(row_t + c * 32, v + c * 32);
    if (R == 16) {
      float t[32];
      tmem_ld32(row_t + DC, t);          // columns past DC + 16 are not used
      tc_wait_ld();
#pragma unroll
      for (int j = 0; j < RU; ++j) u[j] = t[j];
    } else {
#pragma unroll
      for (int c = 0; c < R / 32; ++c) tmem_ld32(row_t + DC + c * 32, u + c * 32);
      tc_wait_ld();
    }
  }
  if (P == 1 && p.ksplit > 1) {
    if (!ok) return;                     // (the split-K path has no cluster barriers)
    float* mine = p.part + (((long long)tile * p.ksplit + ks) * 128 + r) * rowlen;
#pragma unroll
    for (int c = 0; c < DC; c += 4) *reinterpret_cast<float4*>(mine + c) = make_float4(v[c], v[c + 1], v[c + 2], v[c + 3]);
#pragma unroll
    for (int c = 0; c < R; c += 4) *reinterpret_cast<float4*>(mine + DC + c) = make_float4(u[c], u[c + 1], u[c + 2], u[c + 3]);
    __threadfence();
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (et == 0) *last_flag = (atomicAdd(&p.counters[tile], 1) == p.ksplit - 1) ? 1 : 0;
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (*last_flag == 0) return;          // CTA-uniform: another CTA finishes this tile
    __threadfence();
    // every split's partial (this CTA's too), in split order
#pragma unroll
    for (int c = 0; c < DC; ++c) v[c] = 0.f;
#pragma unroll
    for (int c = 0; c < RU; ++c) u[c] = 0.f;
    for (int kk = 0; kk < p.ksplit; ++kk) {
      const float* pk = p.part + (((long long)tile * p.ksplit + kk) * 128 + r) * rowlen;
#pragma unroll
      for (int c = 0; c < DC; c += 4) {
        const float4 o = __ldcg(reinterpret_cast<const float4*>(pk + c));
        v[c] += o.x; v[c + 1] += o.y; v[c + 2] += o.z; v[c + 3] += o.w;
      }
#pragma unroll
      for (int c = 0; c < R; c += 4) {
        const float4 o = __ldcg(reinterpret_cast<const float4*>(pk + DC + c));
        u[c] += o.x; u[c + 1] += o.y; u[c + 2] += o.z; u[c + 3] += o.w;
      }
    }
  }
  if (R > 0 && ok) {
    // U = bf16(s * u) as a K-major tile [R/8][128 rows][8] in the idle stage ring,
    // then one MMA per 16 of R: LoRA update (TMEM at LUP_COL) = U B_h^T
#pragma unroll
    for (int g = 0; g < R / 8; ++g) {
      uint32_t w[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int j0 = g * 8 + 2 * e;
        w[e] = pack_bf16(j0 < p.r ? p.s * u[j0] : 0.f, j0 + 1 < p.r ? p.s * u[j0 + 1] : 0.f);
      }
      st_shared_v4(sbase + g * 2048 + r * 16, w[0], w[1], w[2], w[3]);
    }
    fence_proxy_async_smem();
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (et == 0) {
      if (mbar_wait(bar(QB_LORA), 0, abort_flag, p.wait_limit, p.status)) {
        tc_fence_after();
        constexpr uint32_t idesc = idesc_bf16_f32(128, DC, 0, 0);
#pragma unroll
        for (int kk = 0; kk < R / 16; ++kk)
          umma_bf16(tmem + L::LUP_COL, sdesc_noswz(sbase + kk * 2 * 2048, 2048, 128),
                    sdesc_noswz(sbase + L::B_OFF + kk * 2 * (DC * 16), DC * 16, 128), idesc, kk > 0 ? 1u : 0u);
        umma_commit(bar(QB_LUP));
      } else {
        mbar_arrive(bar(QB_LUP));       // never issued: release the waiters (status already TIMEOUT)
      }
    }
    warp_wait(bar(QB_LUP), 0, abort_flag, p.wait_limit, p.status);
    tc_fence_after();
#pragma unroll
    for (int c = 0; c < DC / 32; ++c) {
      float t[32];
      tmem_ld32(row_t + L::LUP_COL + c * 32, t);
      tc_wait_ld();
#pragma unroll
      for (int k = 0; k < 32; ++k) v[c * 32 + k] += t[k];
    }
  }
  // RMSNorm * w, RoPE on pairs (j, j + D/2), bf16 store; rows past M store
  // nothing; V (K/V mode) is stored as projected
  const bool row_ok = m < p.M;
  const int mr = row_ok ? m : p.M - 1;
  if (!is_v) {
    float ss = 0.f;
    if (ok) {
#pragma unroll
      for (int j = 0; j < DC; ++j) ss = fmaf(v[j], v[j], ss);
    }
    if constexpr (P > 1) {
      // the head's sum of squares: this CTA's columns plus the peers', in part order
      float* red = reinterpret_cast<float*>(smem + L::RED_OFF);
      red[r] = ss;
      cluster_sync_all();   // 1: every part's partial sums are in place
      float tot = 0.f;
#pragma unroll
      for (int pp = 0; pp < P; ++pp) tot += (pp == part) ? ss : ld_dsmem(dsmem_addr(smem_u32(red + r), pp));
      cluster_sync_all();   // 2: no CTA leaves while a peer may still read its sums
      ss = tot;
    }
    const float rinv = rsqrtf(ss * (1.0f / D) + p.eps);
#pragma unroll
    for (int c = 0; c < DC / 2; ++c) {
      const int j = j0 + c;
      const float2 cs = p.rope[(long long)j * p.M + mr];
      const float a = v[c] * rinv * __bfloat162float(p.qnorm_w[j]);
      const float b = v[c + DC / 2] * rinv * __bfloat162float(p.qnorm_w[j + D / 2]);
      v[c] = a * cs.x - b * cs.y;
      v[c + DC / 2] = b * cs.x + a * cs.y;
    }
  } else if constexpr (P > 1) {
    cluster_sync_all();     // V heads: the same two cluster barriers, nothing to exchange
    cluster_sync_all();
  }
  if (ok && row_ok) {
    const long long t = (long long)(m / p.S) * p.S_out + (p.S_out - p.S) + m % p.S;   // output token row
    __nv_bfloat16* base = is_v ? p.out2 : p.q_out;
    __nv_bfloat16* orow = base + (t * p.Hout + head) * D;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      uint4* dst = reinterpret_cast<uint4*>(orow + h * (D / 2) + j0);
      const float* src = v + h * (DC / 2);
#pragma unroll
      for (int c = 0; c < DC / 16; ++c)
        dst[c] = make_uint4(pack_bf16(src[8 * c], src[8 * c + 1]), pack_bf16(src[8 * c + 2], src[8 * c + 3]),
                            pack_bf16(src[8 * c + 4], src[8 * c + 5]), pack_bf16(src[8 * c + 6], src[8 * c + 7]));
    }
  }
}

template <int D, int P>
__global__ void __launch_bounds__(192, 1) qproj_kernel(const __grid_constant__ QprojParams p) {
  using L = QpLayout<D>;
  constexpr int DC = D / P;   // output columns of this CTA (two halves of DC/2)
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR_OFF);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::BAR_OFF + 384);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 392);
  volatile int* last_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 396);
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  const int B_FULL = QB_FULL, B_EMPTY = QB_FULL + L::NS;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  // blockIdx.x = (head * P + part) * ksplit + ks  (P > 1 only with ksplit = 1)
  const int head = blockIdx.x / (P * p.ksplit);
  const int part = (blockIdx.x / p.ksplit) % P;
  const int ks = blockIdx.x % p.ksplit;
  const int tile = blockIdx.y * p.Hq + head;
  const int m0 = blockIdx.y * 128;
  const bool is_v = p.kv && head >= p.Hout;             // K/V mode: this CTA projects V
  const int oh = is_v ? head - p.Hout : head;            // head within its output
  const CUtensorMap* tm_w = is_v ? &p.tm_w2 : &p.tm_w;
  // W rows of this CTA's columns: n0 + j0 + [0, DC/2) and n0 + D/2 + j0 + [0, DC/2)
  const int n0 = oh * D, j0 = part * (DC / 2);
  const int nk = p.hidden / 64;
  const int kb0 = ks * nk / p.ksplit, kb1 = (ks + 1) * nk / p.ksplit;
  const bool lora = p.n_lora > 0;
  const int nmma = DC + (lora ? p.n_lora : 0);            // N of the main MMA
  const uint32_t a_off = L::X_BYTES + DC * 128;           // A rows right below this CTA's W rows
  const uint32_t stage_tx = L::X_BYTES + DC * 128 + (lora ? p.n_lora * 128 : 0);

  if (threadIdx.x == 0) {
    for (int i = 0; i < QB_FULL + 2 * L::NS; ++i) mbar_init(bar(i), 1);
    *abort_flag = 0;
    *last_flag = 0;
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
        // B_h rows of this CTA's columns: r/8 boxes of [DC/2 rows][8 columns] per
        // half (columns past r read as zeros)
        mbar_expect_tx(bar(QB_LORA), (p.n_lora / 8) * DC * 16);
        for (int g = 0; g < p.n_lora / 8; ++g)
          for (int h = 0; h < 2; ++h)
            tma_load_2d(sbase + L::B_OFF + g * DC * 16 + h * (DC / 2) * 16, &p.tm_b, bar(QB_LORA), g * 8,
                        n0 + h * (D / 2) + j0);
      }
      int issued = 0;
      for (int kb = kb0; kb < kb1; ++kb) {
        const int it = kb - kb0, st = it % L::NS;
        if (it >= L::NS &&
            !mbar_wait(bar(B_EMPTY + st), ((it / L::NS) - 1) & 1, abort_flag, p.wait_limit, p.status))
          break;
        const uint32_t x_dst = sbase + st * L::STAGE;
        mbar_expect_tx(bar(B_FULL + st), stage_tx);
        tma_load_2d(x_dst, &p.tm_x, bar(B_FULL + st), kb * 64, m0);
        tma_load_2d(x_dst + L::X_BYTES, tm_w, bar(B_FULL + st), kb * 64, n0 + j0);
        tma_load_2d(x_dst + L::X_BYTES + (DC / 2) * 128, tm_w, bar(B_FULL + st), kb * 64, n0 + D / 2 + j0);
        if (lora) tma_load_2d(x_dst + a_off, &p.tm_a, bar(B_FULL + st), kb * 64, 0);
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
        const uint32_t x_s = sbase + st * L::STAGE;
        const uint32_t w_s = x_s + L::X_BYTES;
#pragma unroll
        for (int k = 0; k < 4; ++k)
          umma_bf16(tmem, sdesc_sw128(x_s + k * 32, 16, 1024), sdesc_sw128(w_s + k * 32, 16, 1024), idesc,
                    (it > 0 || k > 0) ? 1u : 0u);
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
    // and the split-K counters come from the prep kernel just before this one.
    grid_dep_wait();
    const bool acc_ok = warp_wait(bar(QB_ACC), 0, abort_flag, p.wait_limit, p.status);
    // one answer for all four warps: a warp that gave up raised the abort flag
    asm volatile("bar.sync 1, 128;" ::: "memory");
    const bool ok = acc_ok && *abort_flag == 0;
    if (ok) tc_fence_after();
    const int nl = lora ? p.n_lora : 0;
    if (nl == 0)
      qproj_epilogue<D, P, 0>(p, smem, tmem, bars, abort_flag, last_flag, oh, part, is_v, ks, tile, m0, ok);
    else if (nl <= 16)
      qproj_epilogue<D, P, 16>(p, smem, tmem, bars, abort_flag, last_flag, oh, part, is_v, ks, tile, m0, ok);
    else if (nl <= 32)
      qproj_epilogue<D, P, 32>(p, smem, tmem, bars, abort_flag, last_flag, oh, part, is_v, ks, tile, m0, ok);
    else
      qproj_epilogue<D, P, 64>(p, smem, tmem, bars, abort_flag, last_flag, oh, part, is_v, ks, tile, m0, ok);
  }
  if (P > 1 && warp < 2) {
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

template <int D, int P>
static cudaError_t launch_qproj_t(const QprojParams& p, cudaStream_t st) {
  using L = QpLayout<D>;
  cudaError_t e = cudaFuncSetAttribute(qproj_kernel<D, P>, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM);
  if (e != cudaSuccess) return e;
  dim3 grid(p.Hq * P * p.ksplit, (p.M + 127) / 128);
  return launch_pdl(qproj_kernel<D, P>, grid, dim3(192), (size_t)L::SMEM, st, P > 1 ? P : 0, p);
}

cudaError_t launch_qproj(const QprojParams& p, int D, cudaStream_t st) {
  if (p.parts > 1 && p.ksplit > 1) return cudaErrorInvalidValue;
  if (D == 128) {
    if (p.parts == 4) return launch_qproj_t<128, 4>(p, st);
    if (p.parts == 2) return launch_qproj_t<128, 2>(p, st);
    if (p.parts == 1) return launch_qproj_t<128, 1>(p, st);
  }
  if (D == 64) {
    if (p.parts == 2) return launch_qproj_t<64, 2>(p, st);
    if (p.parts == 1) return launch_qproj_t<64, 1>(p, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace att
