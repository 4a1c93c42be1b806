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

// One launch, three independent jobs selected by block index:
//   [0, nb_lora)            one warp per (query row, 4 LoRA outputs): u = s * (A x)
//   [nb_lora, +nb_rope)     one thread per (query row, rotary pair): cos/sin table
//   [.., +nb_b)             one thread per 16 bytes of b_pad
__global__ void __launch_bounds__(256) prep_kernel(const __grid_constant__ PrepParams p, int nb_lora,
                                                   int nb_rope) {
  const int bid = blockIdx.x;
  if (bid < nb_lora) {
    const int warp = (bid * 256 + (int)threadIdx.x) >> 5, lane = threadIdx.x & 31;
    const int groups = 16;                       // 64 padded columns / 4 per warp
    const int m = warp / groups, jg = warp % groups;
    if (m >= p.M) return;
    const int j0 = jg * 4;
    if (j0 >= p.r) {                             // zero padding columns r..63
      if (lane < 4) p.u_pad[(long long)m * 64 + j0 + lane] = __float2bfloat16_rn(0.f);
      return;
    }
    const __nv_bfloat16* xr = p.x + (long long)m * p.hidden;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 2
    for (int k = lane * 8; k < p.hidden; k += 256) {
      float xf[8];
      bf16x8_to_f32(*reinterpret_cast<const uint4*>(xr + k), xf);
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        float af[8];
        bf16x8_to_f32(*reinterpret_cast<const uint4*>(p.lora_a + (long long)(j0 + jj) * p.hidden + k), af);
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[jj] = fmaf(af[e], xf[e], acc[jj]);
      }
    }
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc[jj] += __shfl_xor_sync(0xffffffffu, acc[jj], o);
    }
    if (lane < 4) {
      float v = lane == 0 ? acc[0] : lane == 1 ? acc[1] : lane == 2 ? acc[2] : acc[3];
      p.u_pad[(long long)m * 64 + j0 + lane] = __float2bfloat16_rn(p.s * v);
    }
    return;
  }
  if (bid < nb_lora + nb_rope) {
    // RoPE angle of (row m, pair j): pos * theta^(-2j/D), pos = T_art(req) + (S_kv - S) + i.
    // Formed and reduced modulo 2*pi in double, then sin/cos in float on |angle| <= pi.
    const int half = p.D / 2;
    const long long idx = (long long)(bid - nb_lora) * 256 + threadIdx.x;
    if (idx >= (long long)p.M * half) return;
    const int m = (int)(idx / half), j = (int)(idx % half);
    const int req = m / p.S, i = m % p.S;
    const long long pos = (long long)p.t_art[req] + (p.S_kv - p.S) + i;
    const double ang = (double)pos * p.inv_freq[j];
    const double k = rint(ang * 0.15915494309189533577);   // 1 / (2 pi)
    const double red = fma(-k, 6.283185307179586232, ang);
    float sn, cs;
    sincosf((float)red, &sn, &cs);
    p.rope[idx] = make_float2(cs, sn);
    return;
  }
  // b_pad[n][0..63] = B[n][0..r-1], zeros beyond
  const long long idx = (long long)(bid - nb_lora - nb_rope) * 256 + threadIdx.x;
  if (idx >= (long long)p.d_q * 8) return;
  const int n = (int)(idx / 8), c = (int)(idx % 8);
  uint4 val = make_uint4(0, 0, 0, 0);
  if (c * 8 < p.r) val = *reinterpret_cast<const uint4*>(p.lora_b + (long long)n * p.r + c * 8);
  *reinterpret_cast<uint4*>(p.b_pad + (long long)n * 64 + c * 8) = val;
}

cudaError_t launch_prep(const PrepParams& p, cudaStream_t st) {
  const bool lora = p.lora_a != nullptr && p.lora_b != nullptr && p.r > 0;
  const int nb_lora = lora ? (p.M * 16 * 32 + 255) / 256 : 0;
  const int nb_rope = (int)(((long long)p.M * (p.D / 2) + 255) / 256);
  const int nb_b = lora ? (p.d_q * 8 + 255) / 256 : 0;
  prep_kernel<<<nb_lora + nb_rope + nb_b, 256, 0, st>>>(p, nb_lora, nb_rope);
  return cudaGetLastError();
}

}  // namespace att
