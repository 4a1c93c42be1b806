// prep.cu - small kernels around the main path:
//   * pool_write: copy one artifact's K/V ([L, Hkv, D], Sec. 2 Eq. full-vs-pic:
//     encoded alone at local positions, never changed afterwards) into its
//     paged pool blocks [block][Hkv][64][D];
//   * prep: the cos/sin table of every query row's RoPE angles (App. A.5
//     position ids of the assembled context);
//   * rotate_keys: keys stored before RoPE rotated to their assembled
//     positions when a plan is assembled (App. C.2, EPIC paragraph).
#include <math.h>

#include <algorithm>

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
  // unused tail slots of the last block read as zeros (see pool_write_host_kernel)
  const int tail = L % kBlockTokens;
  if (tail != 0) {
    const long long nt = (long long)(kBlockTokens - tail) * Hkv * cpr;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < nt;
         i += (long long)gridDim.x * blockDim.x) {
      const int c = (int)(i % cpr);
      const int h = (int)((i / cpr) % Hkv);
      const int slot = tail + (int)(i / ((long long)cpr * Hkv));
      const long long dst = (((long long)(first_block + L / kBlockTokens) * Hkv + h) * kBlockTokens + slot) * cpr + c;
      kpool[dst] = make_uint4(0, 0, 0, 0);
      vpool[dst] = make_uint4(0, 0, 0, 0);
    }
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

// The warm-cache load: one pass over every 16-byte chunk of a batch of host
// artifacts.  Consecutive threads read consecutive chunks of one artifact
// (coalesced reads over the CPU-GPU link); each chunk lands in its pool slot
// [block][h][token % 64][:] as in pool_write_kernel.
__global__ void __launch_bounds__(256) pool_write_host_kernel(const __grid_constant__ HostBatch b,
                                                              uint4* __restrict__ kpool,
                                                              uint4* __restrict__ vpool) {
  const int cpr = b.D / 8;
  const long long total = b.chunk_end[b.n - 1];
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    int a = 0;
    while (b.chunk_end[a] <= i) ++a;                    // n <= 64: a short scan
    const long long li = i - (a > 0 ? b.chunk_end[a - 1] : 0);
    const int c = (int)(li % cpr);
    const long long ph = li / cpr;
    const int h = (int)(ph % b.Hkv);
    const int t = (int)(ph / b.Hkv);
    const long long dst =
        (((long long)(b.first[a] + t / kBlockTokens) * b.Hkv + h) * kBlockTokens + t % kBlockTokens) * cpr + c;
    kpool[dst] = b.k[a][li];
    vpool[dst] = b.v[a][li];
  }
  // zero the unused tail slots of each artifact's last block: the pool may
  // hold an earlier artifact there after attuner_pool_reset, and a masked key
  // still multiplies its V row by 0
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < (long long)b.n * kBlockTokens * b.Hkv * cpr;
       i += (long long)gridDim.x * blockDim.x) {
    const int c = (int)(i % cpr);
    const long long r = i / cpr;
    const int h = (int)(r % b.Hkv);
    const int slot = (int)((r / b.Hkv) % kBlockTokens);
    const int a = (int)(r / ((long long)b.Hkv * kBlockTokens));
    const int tail = b.L[a] % kBlockTokens;
    if (tail == 0 || slot < tail) continue;
    const int blk = b.first[a] + b.L[a] / kBlockTokens;
    const long long dst = (((long long)blk * b.Hkv + h) * kBlockTokens + slot) * cpr + c;
    kpool[dst] = make_uint4(0, 0, 0, 0);
    vpool[dst] = make_uint4(0, 0, 0, 0);
  }
}

cudaError_t launch_pool_write_host(const HostBatch& b, __nv_bfloat16* kpool, __nv_bfloat16* vpool,
                                   int num_sms, cudaStream_t st) {
  const long long total = b.chunk_end[b.n - 1];
  long long grid = (total + 255) / 256;
  if (grid > (long long)num_sms * 8) grid = (long long)num_sms * 8;
  pool_write_host_kernel<<<(int)grid, 256, 0, st>>>(b, reinterpret_cast<uint4*>(kpool),
                                                    reinterpret_cast<uint4*>(vpool));
  return cudaGetLastError();
}

// One thread per (query row, rotary pair): the RoPE angle pos * theta^(-2j/D)
// with pos = T_art(req) + (S_kv - S) + i (App. A.5: positions of the
// assembled context), formed and reduced modulo 2*pi in double, then sin/cos
// in float on |angle| <= pi.
__global__ void __launch_bounds__(256) prep_kernel(const __grid_constant__ PrepParams p) {
  grid_dep_wait();     // the scratch it writes may be memory the previous kernel used
  grid_dep_launch();   // the Q projection may start its main loop now
  const long long idx = (long long)blockIdx.x * 256 + threadIdx.x;
  const int half = p.D / 2;
  if (idx >= (long long)p.M * half) return;
  const int j = (int)(idx / p.M), m = (int)(idx % p.M);   // pair-major: coalesced in the epilogue
  const int req = m / p.S, i = m % p.S;
  const long long pos = online_position(p.plan, req, (p.S_kv - p.S) + i);   // assembled position
  p.rope[(long long)j * p.M + m] = rope_cos_sin(pos, p.inv_freq[j]);
}

// One thread per (slot, token row, group of 8 rotary pairs): the cos/sin of
// its 8 angles once, then for every KV head two 16-byte loads (columns
// j0..j0+7 and their partners j0+D/2..) and two 16-byte stores; consecutive
// threads take consecutive pair groups of a row, so each head's row is read
// and written by D/16 neighbouring threads.
__global__ void __launch_bounds__(256) rotate_keys_kernel(const __grid_constant__ RotateParams p) {
  const int groups = p.D / 16;                          // 8-pair groups per row
  const long long idx = (long long)blockIdx.x * 256 + threadIdx.x;
  if (idx >= (long long)p.n_slots * kBlockTokens * groups) return;
  const int g = (int)(idx % groups);
  const int t = (int)((idx / groups) % kBlockTokens);
  const int s = (int)(idx / ((long long)groups * kBlockTokens));
  const int e = p.blocks[s];
  if (e <= 0) return;                                   // online slot: its keys come from the suffix
  const int valid = e & 127, blk = e >> 7;
  if (blk >= p.pool_blocks || valid < 1 || valid > kBlockTokens) {
    set_status(p.status, ATTUNER_ERR_DEVICE_CHECK);
    return;
  }
  const int cpr = p.D / 8;                              // 16-byte chunks per row
  const int j0 = 8 * g;                                 // first pair of the group
  float2 cs[8];
  if (t < valid) {
#pragma unroll
    for (int k = 0; k < 8; ++k) cs[k] = rope_cos_sin((long long)p.slot_pos[s] + t, p.inv_freq[j0 + k]);
  }
  for (int h = 0; h < p.Hkv; ++h) {
    const long long src = (((long long)blk * p.Hkv + h) * kBlockTokens + t) * cpr;
    const long long dst = (((long long)s * p.Hkv + h) * kBlockTokens + t) * cpr;
    uint4 y1 = make_uint4(0, 0, 0, 0), y2 = make_uint4(0, 0, 0, 0);
    if (t < valid) {
      const uint4 a = p.kpool[src + g], b = p.kpool[src + g + cpr / 2];
      const __nv_bfloat16* x1 = reinterpret_cast<const __nv_bfloat16*>(&a);
      const __nv_bfloat16* x2 = reinterpret_cast<const __nv_bfloat16*>(&b);
      uint32_t* o1 = reinterpret_cast<uint32_t*>(&y1);
      uint32_t* o2 = reinterpret_cast<uint32_t*>(&y2);
#pragma unroll
      for (int k = 0; k < 8; k += 2) {
        const float u0 = __bfloat162float(x1[k]), u1 = __bfloat162float(x1[k + 1]);
        const float v0 = __bfloat162float(x2[k]), v1 = __bfloat162float(x2[k + 1]);
        // rotate-half: (x_j, x_{j+D/2}) -> (x_j c - x_{j+D/2} s, x_{j+D/2} c + x_j s)
        o1[k / 2] = pack_bf16(u0 * cs[k].x - v0 * cs[k].y, u1 * cs[k + 1].x - v1 * cs[k + 1].y);
        o2[k / 2] = pack_bf16(v0 * cs[k].x + u0 * cs[k].y, v1 * cs[k + 1].x + u1 * cs[k + 1].y);
      }
    }
    p.krot[dst + g] = y1;
    p.krot[dst + g + cpr / 2] = y2;
  }
}

cudaError_t launch_rotate_keys(const RotateParams& p, cudaStream_t st) {
  const long long n = (long long)p.n_slots * kBlockTokens * (p.D / 16);
  if (n == 0) return cudaSuccess;
  rotate_keys_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_prep(const PrepParams& p, cudaStream_t st) {
  const long long n = (long long)p.M * (p.D / 2);
  return launch_pdl(prep_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, st, 0, p);
}

}  // namespace att
