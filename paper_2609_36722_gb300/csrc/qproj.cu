// qproj.cu - K1b: the adapted query projection of Sec. 3, Eq.
// (query-adaptation), followed by the model's original query RMSNorm and
// RoPE, as ONE tcgen05 GEMM with a fused epilogue:
//
//   Q[m, h, :] = RoPE( RMSNorm( [x_m | u_m] . [W_q | B]_h^T ) * w, pos_m )
//
// where u = s * (A x) (bf16, from prep.cu).  Concatenating along K turns the
// low-rank update into one more 64-wide K block of the same GEMM (only
// ceil(r/16) of its four 16-wide MMA steps are issued).
//
// CTA tile: 128 query rows x one head (N = D = 64 or 128), so every
// accumulator row holds a whole head and the RMSNorm needs no cross-CTA
// reduction.  Warp 0: TMA producer; warp 1: TMEM owner + MMA issuer; warps
// 2..5: epilogue (one accumulator row per thread, tcgen05.ld 32x32b).
#include "kernels.h"

namespace att {

template <int D>
struct QpLayout {
  static constexpr int NS = (D == 128) ? 6 : 8;
  static constexpr int A_BYTES = 128 * 128;   // 128 rows x 64 bf16
  static constexpr int B_BYTES = D * 128;     // D rows x 64 bf16
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr int BAR_OFF = NS * STAGE;
  static constexpr int SMEM = BAR_OFF + 512 + 1024;   // + alignment slack
  static constexpr uint32_t TMEM_COLS = (D < 32) ? 32 : D;
};

template <int D>
__global__ void __launch_bounds__(192, 1) qproj_kernel(const __grid_constant__ QprojParams p) {
  using L = QpLayout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR_OFF);
  // bars[0..NS): full, bars[NS..2NS): empty, bars[2NS]: accumulator ready, bars[2NS+1]: drain
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::BAR_OFF + 384);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 392);
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  const int B_FULL = 0, B_EMPTY = L::NS, B_ACC = 2 * L::NS, B_DRAIN = 2 * L::NS + 1;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int head = blockIdx.x;
  const int m0 = blockIdx.y * 128;
  const int n0 = head * D;
  const int nk_main = p.hidden / 64;
  const int nk = nk_main + (p.lora_ksteps > 0 ? 1 : 0);

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2 * L::NS + 2; ++i) mbar_init(bar(i), 1);
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
      tma_prefetch_desc(&p.tm_w);
      int issued = 0;
      for (int kb = 0; kb < nk; ++kb) {
        const int st = kb % L::NS;
        if (kb >= L::NS &&
            !mbar_wait(bar(B_EMPTY + st), ((kb / L::NS) - 1) & 1, abort_flag, p.wait_limit, p.status))
          break;
        const uint32_t a_dst = sbase + st * L::STAGE;
        const uint32_t b_dst = a_dst + L::A_BYTES;
        mbar_expect_tx(bar(B_FULL + st), L::STAGE);
        if (kb < nk_main) {
          tma_load_2d(a_dst, &p.tm_x, bar(B_FULL + st), kb * 64, m0);
          tma_load_2d(b_dst, &p.tm_w, bar(B_FULL + st), kb * 64, n0);
        } else {
          tma_load_2d(a_dst, &p.tm_u, bar(B_FULL + st), 0, m0);
          tma_load_2d(b_dst, &p.tm_b, bar(B_FULL + st), 0, n0);
        }
        issued = kb + 1;
      }
      if (*abort_flag) {   // let every copy this CTA issued land before exiting
        for (int kb = (issued > L::NS ? issued - L::NS : 0); kb < issued; ++kb)
          mbar_drain(bar(B_FULL + kb % L::NS), (kb / L::NS) & 1, p.status);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, D, 0, 0);
      bool ok = true;
      bool any = false;
      for (int kb = 0; kb < nk; ++kb) {
        const int st = kb % L::NS;
        if (!mbar_wait(bar(B_FULL + st), (kb / L::NS) & 1, abort_flag, p.wait_limit, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_s = sbase + st * L::STAGE;
        const uint32_t b_s = a_s + L::A_BYTES;
        const int ksteps = (kb < nk_main) ? 4 : p.lora_ksteps;
        for (int k = 0; k < ksteps; ++k) {
          umma_bf16(tmem, sdesc_sw128(a_s + k * 32, 16, 1024), sdesc_sw128(b_s + k * 32, 16, 1024),
                    idesc, (kb > 0 || k > 0) ? 1u : 0u);
          any = true;
        }
        umma_commit(bar(B_EMPTY + st));
      }
      if (ok) {
        umma_commit(bar(B_ACC));
      } else if (any) {
        umma_commit(bar(B_DRAIN));
        mbar_drain(bar(B_DRAIN), 0, p.status);
      }
    }
  } else {
    // epilogue: warps 2..5 -> TMEM lane quadrants 2, 3, 0, 1
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const int m = m0 + r;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    if (warp_wait(bar(B_ACC), 0, abort_flag, p.wait_limit, p.status)) {
      tc_fence_after();
      float v[D];
#pragma unroll
      for (int c = 0; c < D / 32; ++c) tmem_ld32(tmem + lane_base + c * 32, v + c * 32);
      tc_wait_ld();
      if (m < p.M) {
        float ss = 0.f;
#pragma unroll
        for (int j = 0; j < D; ++j) ss = fmaf(v[j], v[j], ss);
        const float rinv = rsqrtf(ss * (1.0f / D) + p.eps);
#pragma unroll
        for (int j = 0; j < D; ++j) v[j] = v[j] * rinv * __bfloat162float(p.qnorm_w[j]);
        const float2* rp = p.rope + (long long)m * (D / 2);
#pragma unroll
        for (int j = 0; j < D / 2; ++j) {
          const float2 cs = rp[j];
          const float a = v[j], b = v[j + D / 2];
          v[j] = a * cs.x - b * cs.y;
          v[j + D / 2] = b * cs.x + a * cs.y;
        }
        uint4* dst = reinterpret_cast<uint4*>(p.q_out + ((long long)m * p.Hq + head) * D);
#pragma unroll
        for (int c = 0; c < D / 8; ++c)
          dst[c] = make_uint4(pack_bf16(v[8 * c], v[8 * c + 1]), pack_bf16(v[8 * c + 2], v[8 * c + 3]),
                              pack_bf16(v[8 * c + 4], v[8 * c + 5]), pack_bf16(v[8 * c + 6], v[8 * c + 7]));
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
static cudaError_t launch_qproj_t(const QprojParams& p, cudaStream_t st) {
  using L = QpLayout<D>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(qproj_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  dim3 grid(p.Hq, (p.M + 127) / 128);
  qproj_kernel<D><<<grid, 192, L::SMEM, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_qproj(const QprojParams& p, int D, cudaStream_t st) {
  if (D == 128) return launch_qproj_t<128>(p, st);
  if (D == 64) return launch_qproj_t<64>(p, st);
  return cudaErrorInvalidValue;
}

}  // namespace att
