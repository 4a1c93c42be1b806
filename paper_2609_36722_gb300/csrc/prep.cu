// prep.cu - small kernels around the main path:
//   * pool_write: copy one artifact's K/V ([L, Hkv, D], Sec. 2 Eq. full-vs-pic:
//     encoded alone at local positions, never changed afterwards) into its
//     paged pool blocks [block][Hkv][64][D];
//   * prep: per query row, the LoRA down-projection u = s * (A x) of
//     Sec. 3 Eq. (query-adaptation), rounded to bf16 and zero-padded to 64
//     columns (one extra K block of the Q-projection GEMM), the cos/sin table
//     of the row's RoPE angles, and B zero-padded to 64 columns.
#include <math.h>

#include "kernels.h"

namespace att {

__global__ void pool_write_kernel(const uint4* __restrict__ k, const uint4* __restrict__ v,
                                  uint4* __restrict__ kpool, uint4* __restrict__ vpool, int L,
                                  int Hkv, int D, int first_block) {
  const int cpr = D / 8;                       // 16-byte chunks per row
  const long long total = (long long)L * Hkv * cpr;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    const int c = (int)(i % cpr);
    const long long ph = i / cpr;
    const int h = (int)(ph % Hkv);
    const int p = (int)(ph / Hkv);
    const long long dst =
        (((long long)(first_block + p / kBlockTokens) * Hkv + h) * kBlockTokens + p % kBlockTokens) *
            cpr + c;
    kpool[dst] = k[i];
    vpool[dst] = v[i];
  }
}

cudaError_t launch_pool_write(const __nv_bfloat16* k, const __nv_bfloat16* v, __nv_bfloat16* kpool,
                              __nv_bfloat16* vpool, int L, int Hkv, int D, int first_block,
                              cudaStream_t st) {
  const long long total = (long long)L * Hkv * (D / 8);
  int grid = (int)((total + 255) / 256);
  if (grid > 152 * 16) grid = 152 * 16;
  pool_write_kernel<<<grid, 256, 0, st>>>(reinterpret_cast<const uint4*>(k),
                                          reinterpret_cast<const uint4*>(v),
                                          reinterpret_cast<uint4*>(kpool),
                                          reinterpret_cast<uint4*>(vpool), L, Hkv, D, first_block);
  return cudaGetLastError();
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4& u, float* f) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 t = __bfloat1622float2(h[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}

// One warp per query row: u_pad row, rope row.  Extra blocks: b_pad.
__global__ void __launch_bounds__(128) prep_kernel(const PrepParams p, int row_blocks) {
  if ((int)blockIdx.x >= row_blocks) {
    // b_pad[n][0..63] = B[n][0..r-1], zeros beyond
    const long long idx = (long long)(blockIdx.x - row_blocks) * blockDim.x + threadIdx.x;
    if (p.lora_b == nullptr || idx >= (long long)p.d_q * 8) return;
    const int n = (int)(idx / 8), c = (int)(idx % 8);
    uint4 val = make_uint4(0, 0, 0, 0);
    if (c * 8 < p.r) val = *reinterpret_cast<const uint4*>(p.lora_b + (long long)n * p.r + c * 8);
    *reinterpret_cast<uint4*>(p.b_pad + (long long)n * 64 + c * 8) = val;
    return;
  }
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int m = blockIdx.x * 4 + warp;
  if (m >= p.M) return;

  if (p.lora_a != nullptr && p.r > 0) {
    float acc[64];
#pragma unroll
    for (int j = 0; j < 64; ++j) acc[j] = 0.f;
    const __nv_bfloat16* xr = p.x + (long long)m * p.hidden;
    for (int k0 = 0; k0 < p.hidden; k0 += 256) {
      const int k = k0 + lane * 8;
      if (k < p.hidden) {
        float xf[8];
        bf16x8_to_f32(*reinterpret_cast<const uint4*>(xr + k), xf);
#pragma unroll
        for (int j = 0; j < 64; ++j) {
          if (j < p.r) {
            float af[8];
            bf16x8_to_f32(*reinterpret_cast<const uint4*>(p.lora_a + (long long)j * p.hidden + k), af);
            float s = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) s = fmaf(af[e], xf[e], s);
            acc[j] += s;
          }
        }
      }
    }
#pragma unroll
    for (int j = 0; j < 64; ++j) {
      if (j < p.r) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[j] += __shfl_xor_sync(0xffffffffu, acc[j], o);
      }
    }
    // lane writes columns 2*lane, 2*lane+1
    float lo = 0.f, hi = 0.f;
#pragma unroll
    for (int j = 0; j < 64; ++j) {
      if (j == 2 * lane) lo = (j < p.r) ? p.s * acc[j] : 0.f;
      if (j == 2 * lane + 1) hi = (j < p.r) ? p.s * acc[j] : 0.f;
    }
    reinterpret_cast<__nv_bfloat162*>(p.u_pad + (long long)m * 64)[lane] =
        __floats2bfloat162_rn(lo, hi);
  }

  // RoPE angles of this row: pos = T_art(req) + (S_kv - S) + i, pairs (j, j + D/2)
  // turned by pos * theta^(-2j/D).  The angle is formed and reduced modulo
  // 2*pi in double, then sin/cos are taken in float on |angle| <= pi.
  const int req = m / p.S, i = m % p.S;
  const long long pos = (long long)p.t_art[req] + (p.S_kv - p.S) + i;
  const int half = p.D / 2;
  const double two_pi = 6.283185307179586476925286766559;
  for (int j = lane; j < half; j += 32) {
    const double inv_freq = pow(p.theta, -2.0 * (double)j / (double)p.D);
    double ang = (double)pos * inv_freq;
    ang -= two_pi * floor(ang / two_pi);
    if (ang > 3.14159265358979323846) ang -= two_pi;
    float sn, cs;
    sincosf((float)ang, &sn, &cs);
    p.rope[(long long)m * half + j] = make_float2(cs, sn);
  }
}

cudaError_t launch_prep(const PrepParams& p, cudaStream_t st) {
  const int row_blocks = (p.M + 3) / 4;
  const int b_blocks = (p.lora_b != nullptr && p.r > 0) ? (p.d_q * 8 + 127) / 128 : 0;
  prep_kernel<<<row_blocks + b_blocks, 128, 0, st>>>(p, row_blocks);
  return cudaGetLastError();
}

}  // namespace att
