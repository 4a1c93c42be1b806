// common.cuh - device-side building blocks shared by the kernels of
// libattuner: inline-PTX wrappers for mbarriers, TMA (cp.async.bulk.tensor),
// tcgen05 (UMMA issue, TMEM alloc/ld/st, commit) and warp MMA, bounded
// waits that report a status instead of hanging, and the launch parameter
// structs.  sm_103a only.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/attuner.h"
#include "plan.h"

#define ATT_DEV __device__ __forceinline__

namespace att {

// Plan arrays on the device.
// A request's virtual block list ("slots"): its artifact blocks in prompt
// order (entry > 0: pool_block << 7 | valid tokens), held by the plan, then
// chunks of 64 online rows (entry < 0: -((online row0 << 7 | rows) + 1)),
// appended by the kernels: every online row 0 .. S_kv - 1 of the request (the
// explicit spans of a prompt layout, then the final span, the suffix).  An
// online span between artifacts therefore takes no slot of its own: online
// keys are visible by online row (online rows are in assembled order), and
// artifact slots by the span a query sits in.
struct PlanDev {
  const int32_t* blk_off;   // [n_req + 1] CSR offsets into blocks
  const int32_t* blocks;    // slot entries as above
  const int32_t* t_art;     // [n_req] artifact tokens
  const int32_t* o_rows;    // [n_req] online rows in the plan's explicit spans
  const int32_t* span_off;  // [n_req + 1] CSR offsets into spans
  const int4* spans;        // explicit online spans: (online row0, rows, artifact slots before, artifact tokens before)
  // artifact references and their grouping by artifact (PlanTables)
  const int32_t* req_art_off;   // [n_req + 1] CSR offsets into the references
  const int32_t* ref_nblk;      // blocks of each reference (plan order)
  const int32_t* dist_off;      // [n_dist + 1] references of each distinct artifact
  const int32_t* dist_src;      // [n_dist] plan slot of its first reference's first block
  const int32_t* dist_nb;       // [n_dist] its blocks
  const int32_t* dref_req;      // per reference in grouping order: its request,
  const int32_t* dref_j;        //   its ordinal among the request's references,
  const int32_t* dref_nref;     //   and the request's number of references
  int32_t pool_blocks;      // capacity, for bounds checks
  int32_t has_spans;        // 0: no request has explicit online spans (o_rows all 0; no loads needed)
};

ATT_DEV int plan_o_rows(const PlanDev& pl, int req) { return pl.has_spans ? pl.o_rows[req] : 0; }

ATT_DEV int online_entry(int row0, int rows) { return -(((row0 << 7) | rows) + 1); }
ATT_DEV int slot_row0(int e) { return (-e - 1) >> 7; }   // online slots only

// Artifact slots that a query at online row t of request `req` sees: those
// before its span in the prompt (all nab of them for rows of the final span).
// It sees online rows 0 .. t, i.e. the keys of slots nab .. nab + t/64 up to
// its own row.
ATT_DEV int art_slots_seen(const PlanDev& pl, int req, int t, int nab) {
  if (t >= plan_o_rows(pl, req)) return nab;
  for (int k = pl.span_off[req]; k < pl.span_off[req + 1]; ++k) {
    const int4 sp = pl.spans[k];
    if (t < sp.x + sp.y) return sp.z;
  }
  return 0;   // not reached for a valid plan
}
// assembled position of online row t (App. A.5 position ids)
ATT_DEV int online_position(const PlanDev& pl, int req, int t) {
  const int o = plan_o_rows(pl, req);
  if (t >= o) return pl.t_art[req] + t;
  for (int k = pl.span_off[req]; k < pl.span_off[req + 1]; ++k) {
    const int4 sp = pl.spans[k];
    if (t < sp.x + sp.y) return sp.w + t;
  }
  return t;   // not reached for a valid plan
}

// cos and sin of the RoPE angle pos * inv_freq: the angle formed and reduced
// modulo 2 pi in double (positions reach 2^22 and more), then sin / cos in
// float on |angle| <= pi.
ATT_DEV float2 rope_cos_sin(long long pos, double inv_freq) {
  const double ang = (double)pos * inv_freq;
  const double k = rint(ang * 0.15915494309189533577);   // 1 / (2 pi)
  const double red = fma(-k, 6.283185307179586232, ang);
  float sn, cs;
  sincosf((float)red, &sn, &cs);
  return make_float2(cs, sn);
}

ATT_DEV int find_req(const WorkTable& w, int cta) {
  int lo = 0, hi = w.n_req - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (w.base[mid] <= cta) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// ---------------------------------------------------------------------------
// Status word (device): first error wins.
// ---------------------------------------------------------------------------
ATT_DEV void set_status(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

ATT_DEV uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---------------------------------------------------------------------------
// mbarrier
// ---------------------------------------------------------------------------
ATT_DEV void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
ATT_DEV void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
ATT_DEV void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
ATT_DEV void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
ATT_DEV bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait.  Returns true once the phase with `parity` has completed.
// Returns false when *abort became non-zero (another role gave up) or when
// `limit` clock cycles passed; in the latter case it raises the abort flag
// and records ATTUNER_ERR_TIMEOUT in the status word.
ATT_DEV bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort, long long limit,
                       int* status) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (*abort) return false;
    if (clock64() - t0 > limit) {
      *abort = 1;
      set_status(status, ATTUNER_ERR_TIMEOUT);
      return false;
    }
  }
}

// Warp-uniform form of mbar_wait: every lane of the warp waits and all lanes
// get the same answer, so a timeout never splits a warp in front of a
// .sync.aligned instruction.
ATT_DEV bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort, long long limit,
                       int* status) {
  const bool r = mbar_wait(bar, parity, abort, limit, status);
  return __all_sync(0xffffffffu, r);
}

// Drain wait used on the abort path: waits for work this CTA itself issued
// (TMA copies, MMAs), or copies that peers issue unconditionally, which
// complete without any other role's help.  False after a timeout.
constexpr long long kDrainLimit = 1ll << 32;   // ~2 s at 2 GHz
ATT_DEV bool mbar_drain(uint32_t bar, uint32_t parity, int* status) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kDrainLimit) { set_status(status, ATTUNER_ERR_TIMEOUT); return false; }
  }
  return true;
}

// ---------------------------------------------------------------------------
// TMA (tiled tensor copies global -> shared, completion on an mbarrier)
// ---------------------------------------------------------------------------
ATT_DEV void tma_prefetch_desc(const CUtensorMap* m) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(m)) : "memory");
}
ATT_DEV void tma_load_2d(uint32_t dst, const CUtensorMap* m, uint32_t bar, int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), "r"(c0), "r"(c1)
      : "memory");
}
ATT_DEV void tma_load_4d(uint32_t dst, const CUtensorMap* m, uint32_t bar, int c0, int c1, int c2,
                         int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
      : "memory");
}
ATT_DEV void tma_load_5d(uint32_t dst, const CUtensorMap* m, uint32_t bar, int c0, int c1, int c2,
                         int c3, int c4) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6, %7}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4)
      : "memory");
}

// tiled tensor store shared -> global (bulk group of the issuing thread); boxes
// past the tensor's bounds are clipped.  Coordinates must not be negative.
ATT_DEV void tma_store_4d(const CUtensorMap* m, uint32_t src, int c0, int c1, int c2, int c3) {
  asm volatile("cp.async.bulk.tensor.4d.global.shared::cta.tile.bulk_group [%0, {%2, %3, %4, %5}], [%1];"
               ::"l"(reinterpret_cast<uint64_t>(m)), "r"(src), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
               : "memory");
}
// waits until the bulk copies of this thread have read their shared-memory source
ATT_DEV void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }

// generic-proxy shared-memory writes -> visible to the async proxy (UMMA, TMA)
ATT_DEV void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// the same, both directions, for every state space (global included)
ATT_DEV void fence_proxy_async_all() {
  asm volatile("fence.proxy.async;" ::: "memory");
}

// Untiled bulk copies (cp.async.bulk): both addresses 16-byte aligned and the
// size a multiple of 16.  A load completes on an mbarrier (complete_tx); stores
// are tracked per thread in bulk groups.
ATT_DEV void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(dst), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
               : "memory");
}
ATT_DEV void bulk_store(void* dst, uint32_t src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;"
               ::"l"(reinterpret_cast<uint64_t>(dst)), "r"(src), "r"(bytes)
               : "memory");
}
ATT_DEV void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// waits until every committed bulk store of this thread has been performed
ATT_DEV void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// ---------------------------------------------------------------------------
// Programmatic dependent launch.  Kernels of this library are launched so
// that they may start while the previous kernel in the stream is finishing.
// A kernel calls grid_dep_wait() before it reads anything an earlier kernel
// of the stream may still be writing, and before its first global write;
// once the previous grid has completed it returns at once.
// grid_dep_launch() lets the next kernel start its own prologue early.
// ---------------------------------------------------------------------------
ATT_DEV void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
ATT_DEV void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ---------------------------------------------------------------------------
// Thread-block clusters: barrier and distributed shared memory
// ---------------------------------------------------------------------------
// every thread of every CTA in the cluster; release/acquire orders the shared
// memory writes before it with the peers' reads after it
ATT_DEV void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// shared::cluster address of the same offset in the shared memory of CTA `rank`
ATT_DEV uint32_t dsmem_addr(uint32_t saddr, uint32_t rank) {
  uint32_t d;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(saddr), "r"(rank));
  return d;
}
ATT_DEV float ld_dsmem(uint32_t caddr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(caddr) : "memory");
  return v;
}
// bulk copy of `bytes` from this CTA's shared memory into a peer's (both
// addresses 16-byte aligned, size a multiple of 16); completes on the peer's
// mbarrier `cbar` (a shared::cluster address)
ATT_DEV void bulk_push_dsmem(uint32_t cdst, uint32_t src, uint32_t bytes, uint32_t cbar) {
  asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(cdst), "r"(src), "r"(bytes), "r"(cbar)
               : "memory");
}

// ---------------------------------------------------------------------------
// tcgen05: tensor memory and the 5th-generation MMA (cta_group::1)
// ---------------------------------------------------------------------------
ATT_DEV void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
}
ATT_DEV void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
ATT_DEV void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
ATT_DEV void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
ATT_DEV void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
ATT_DEV void tc_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
ATT_DEV void tc_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// D[tmem] (+)= A[smem desc] * B[smem desc], kind::f16 (bf16 in, fp32 accumulate)
ATT_DEV void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                       uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// mbarrier arrives once all tcgen05 operations issued so far by this thread complete
ATT_DEV void umma_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

// Shared-memory matrix descriptor, 128-byte swizzle (tcgen05 format):
// start>>4 in [0,14), leading byte offset>>4 in [16,30), stride byte
// offset>>4 in [32,46), version 1 at bit 46, layout SWIZZLE_128B (2) in [61,64).
ATT_DEV uint64_t sdesc_sw128(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor, kind::f16: D fp32, A/B bf16, dense.
// a_mn / b_mn select MN-major operands; N>>3 at bit 17, M>>4 at bit 24.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N, int a_mn, int b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)a_mn << 15) | ((uint32_t)b_mn << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// 32 lanes x 32 consecutive 32-bit columns: thread i of the warp receives
// lane (warp_quadrant*32 + i), columns col..col+31.
ATT_DEV void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t* r = reinterpret_cast<uint32_t*>(v);
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}
ATT_DEV void tmem_st32(uint32_t taddr, const float* v) {
  const uint32_t* r = reinterpret_cast<const uint32_t*>(v);
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

// ---------------------------------------------------------------------------
// small math helpers
// ---------------------------------------------------------------------------
ATT_DEV float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
ATT_DEV float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
// packed fp32 pairs (two lanes of the FMA pipe per instruction)
ATT_DEV uint64_t f2_pack(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
ATT_DEV void f2_unpack(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
ATT_DEV uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
ATT_DEV uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
ATT_DEV uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
ATT_DEV void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c),
               "r"(d)
               : "memory");
}

// Warp MMA m16n8k16 bf16 -> fp32 (legacy tensor path; used by the HBM-bound
// decode kernel where the tensor work is far below the memory time).
ATT_DEV void mma_16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
ATT_DEV void ldmatrix_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
ATT_DEV void ldmatrix_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                               uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// Byte offset of 16-byte chunk `chunk` (0..7) of row `row` inside a tile of
// 128-byte rows written by TMA with CU_TENSOR_MAP_SWIZZLE_128B (tile base
// 1024-byte aligned): the chunk index is XORed with row % 8.
ATT_DEV uint32_t sw128_off(int row, int chunk) {
  return (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

}  // namespace att
