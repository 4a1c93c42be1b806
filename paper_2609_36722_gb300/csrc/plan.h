// plan.h - host-only planning of the attention path (plain C++, no CUDA):
// the block table of an assembled request list and the split-KV decomposition
// of one attention launch.  Compiled into libattuner and, on its own, into the
// CPU tests of this logic.
#pragma once

#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/attuner.h"

// functions that the kernels use too (plain inline C++ for the host-only build)
#ifdef __CUDACC__
#define ATT_HD __host__ __device__ __forceinline__
#else
#define ATT_HD inline
#endif

namespace att {

constexpr int kBlockTokens = ATTUNER_BLOCK_TOKENS;   // 64 tokens per paged block
constexpr int kMaxReq = 512;                         // requests per launch (kernel-param tables)

// rows per CTA of each attention kernel
constexpr int kTcRows = 256;      // packed query rows per CTA of attn_tc (two tiles)
constexpr int kTcTileRows = 128;  // rows per query tile (one MMA M)
constexpr int kMmaRows = 16;
// largest split chunk (virtual blocks) the kernels' shared-memory block list holds
constexpr int kMaxChunkBlocks = 4096;
// the warp-MMA kernel's list is shorter, so that two of its CTAs share an SM
constexpr int kMmaMaxChunkBlocks = 1024;
// most split-KV chunks of one (request, KV head, row tile) in the tcgen05 kernel
constexpr int kMaxSplits = 32;
// most distinct artifacts of a launch whose reads are shared (WorkTable::nsplit
// holds one unit offset per distinct artifact and the total)
constexpr int kMaxShareArts = kMaxReq - 1;

// ---------------------------------------------------------------------------
// The Q-projection kernel's shared-memory geometry (qproj.cuh), which the
// host's choice of its launch shape obeys too.  A stage of the TMA ring holds
// MR x tiles (128 rows x 64 bf16), the head's D rows of W_q and up to 64 rows
// of LoRA A; the ring takes as many stages as fit in 200 KiB.  With the K
// dimension split over a cluster, the fp32 partial rows of the tile (D + R
// columns, R = LoRA rank rounded up to 16) are exchanged in the ring, at a row
// pitch that is 4 mod 8 floats.
ATT_HD constexpr int qp_stage_bytes(int D, int MR) { return MR * 128 * 128 + D * 128 + 64 * 128; }
ATT_HD constexpr int qp_ring_bytes(int D, int MR) {
  return (200 * 1024) / qp_stage_bytes(D, MR) * qp_stage_bytes(D, MR);
}
ATT_HD constexpr int qp_pitch(int W) { return W + ((12 - W % 8) % 8); }
ATT_HD constexpr int qp_recv_bytes(int MR, int D, int R) { return MR * 128 * qp_pitch(D + R) * 4; }
ATT_HD constexpr int qp_lora_width(int n_lora) {
  return n_lora == 0 ? 0 : (n_lora <= 16 ? 16 : (n_lora <= 32 ? 32 : 64));
}

// Launch shapes of the projection kernel: mr = 1 or 2 accumulators of 128
// rows per CTA, ks = 1, 2, 4 or 8 CTAs (a cluster) splitting the K dimension
// of a tile.  Supported where the K-split epilogue keeps at least 8 rotary
// pairs per thread (ks/mr threads per row) and the exchange fits the ring.
bool qproj_shape_supported(int D, int mr, int ks, int n_lora);

struct QpPolicy {
  int32_t head_dim, hidden, num_sms;
  int32_t opt_rows;    // 128 or 256 pins the rows per CTA, 0 = chosen here
  int32_t opt_split;   // 1, 2, 4 or 8 pins the K slices, 0 = chosen here
};
struct QpShape {
  int mr, ks;          // {0, 0}: no supported shape under the options
};
// The shape for `heads` heads (grid heads: 2 Hkv in K/V mode) and M rows,
// LoRA rank rounded up to 16 (n_lora, 0 without an adapter).
QpShape choose_qproj_shape(const QpPolicy& pol, int heads, int M, int n_lora);

// ---------------------------------------------------------------------------
// Work decomposition shared by the attention kernels (passed by value).
// A request's KV sequence is a list of "virtual blocks": its artifact blocks
// (from the plan's block table, runtime order) followed by ceil(S_kv/64)
// suffix chunks.  Each CTA owns one (request, kv head, row tile) and a
// contiguous range of virtual blocks (one split-KV chunk).
// CTA index = base[req] + (split * n_kv_heads + kv_head) * row_tiles + row_tile
//
// Shared reads (warp-MMA kernel, share = 1): when several requests use the
// same artifact, one CTA reads a chunk of it for up to `members` requests
// (members x S x G <= 16 packed rows) instead of each request reading it on
// its own.  Work units per KV head: first the artifact units - distinct
// artifact d (the plan's dist_* tables) in chunks of chunk_blocks of its
// blocks, times groups of `members` of its references - numbered from
// nsplit[d] (nsplit[n_dist] = art_units), then suffix units: request r's
// chunks of online rows, art_units + r * suf_chunks + chunk.  CTA index:
// artifact unit u of KV head h at h * art_units + u, then the suffix units of
// every head, unit art_units + v of head h at Hkv * art_units + h * n_req *
// suf_chunks + v (the short suffix CTAs last).  Every (reference, chunk) and every
// suffix chunk leaves a partial result of its request; request r's partials
// are records base[r] .. base[r] + P_r - 1 (the references' chunks in prompt
// order, then the suffix chunks), n_part in all per KV head, and the last
// CTA to finish one of them merges the request's P_r partials in that order.
// ---------------------------------------------------------------------------
struct WorkTable {
  int32_t n_req;
  int32_t row_tiles;      // row tiles per (request, kv head)
  int32_t chunk_blocks;   // virtual blocks per split
  int32_t n_cta;
  // tcgen05 kernel only: 0 = splits of a row tile are independent CTAs merged
  // through global memory; > 0 = every row tile has exactly this many splits,
  // launched as one thread-block cluster (split = rank in the cluster) and
  // merged through distributed shared memory.
  int32_t cluster;
  int32_t base[kMaxReq];
  int32_t nsplit[kMaxReq];
  // shared reads (see above); share = 0 for the per-request decomposition
  int32_t share;
  int32_t members;        // requests per CTA
  int32_t n_dist;         // distinct artifacts
  int32_t art_units;      // artifact units per KV head
  int32_t suf_chunks;     // suffix units of each request
  int32_t n_part;         // partial records per KV head
  int32_t whole_refs;     // every artifact fits one chunk: a reference's partial index is its ordinal
};

// A registered artifact: ceil(L/64) consecutive pool blocks from first_block
// (local token p in block first_block + p/64, row p%64).
struct Artifact {
  int32_t first_block;
  int32_t L;
  int32_t n_blocks;
};

// The host side of an assembled plan.  Items >= 0 given to assembly are
// artifact ids; items < 0 (prompt layouts only) are online spans of -item rows.
struct PlanTables {
  int32_t n_req = 0;
  std::vector<int32_t> req_off;       // CSR over the items given to assembly
  std::vector<int32_t> req_art_off;   // CSR over art_ids
  std::vector<int32_t> art_ids;       // artifact ids in prompt order
  std::vector<Artifact> art_used;     // their registry entries (the plan's own copy)
  std::vector<int32_t> blk_off;       // CSR over blocks
  // artifact slots in prompt order: pool_block << 7 | valid tokens (> 0).
  // Online spans take no slot: a launch reads every online row of a request
  // (explicit spans and the final span, in online-row order) as 64-row chunks
  // after the artifact slots.
  std::vector<int32_t> blocks;
  std::vector<int32_t> t_art;         // artifact tokens of each request
  std::vector<int32_t> o_rows;        // online rows of each request's explicit spans
  std::vector<int32_t> span_off;      // CSR over spans
  std::vector<int32_t> spans;         // 4 per span: online row0, rows, artifact slots before, artifact tokens before
  int32_t max_o_rows = 0;
  // artifact references (one per art_ids entry, CSR by req_art_off): the
  // request, the slot of its first block in the request's slot list and its
  // block count; and the references of each distinct artifact id (ascending
  // id, references in plan order within one id), CSR by dist_off
  std::vector<int32_t> ref_req, ref_slot, ref_nblk;
  std::vector<int32_t> dist_off;      // [n_dist + 1]
  std::vector<int32_t> dist_refs;
  // what the decode kernel reads of them, flattened so that one load (two for
  // the blocks) reaches it: per distinct artifact the plan slot of its first
  // reference's first block and its block count; per reference in dist_refs
  // order its request, its ordinal among that request's references and the
  // request's number of references
  std::vector<int32_t> dist_src, dist_nb;
  std::vector<int32_t> dref_req, dref_j, dref_nref;
  int n_dist() const { return dist_off.empty() ? 0 : (int)dist_off.size() - 1; }
};

// Fills `t` from the request lists (items[offs[r] .. offs[r+1]) of request r)
// against the registry `arts`.  Returns ATTUNER_OK, or an error status with
// `err` set and `t` unspecified.
attuner_status build_plan_tables(const std::vector<Artifact>& arts, const int32_t* items, const int32_t* offs,
                                 int32_t n_req, bool layout, PlanTables& t, std::string& err);

// The artifact blocks and the token index map of a plan, as the public
// attuner_plan_export describes them (sizes_inout: capacities in, counts out).
attuner_status export_plan_tables(const PlanTables& t, int32_t* block_table, int32_t* valid_len,
                                  int32_t* index_map, int32_t* token_art, int32_t* token_off, int64_t* sizes,
                                  std::string& err);

// What the split-KV choice depends on besides the plan.
struct SplitPolicy {
  int32_t n_q_heads, n_kv_heads;
  int32_t num_sms;
  int32_t opt_split;          // virtual blocks per chunk, 0 = chosen here
  int32_t opt_merge;          // 0 = chosen here, 1 = through global memory, 2 = cluster
  int32_t tc_clusters[9];     // co-resident clusters of n tcgen05 CTAs (n = 2, 4)
  // which slots of each request the launch reads: 0 every slot, 1 the plan's
  // artifact slots only, 2 the chunks of the online rows only (for a plan
  // without online spans: the suffix)
  int32_t kv_part = 0;
  // shared reads of the warp-MMA kernel: 0 where they save 10 % or more of
  // the block reads, 1 never, 2 wherever they apply (every query sees every
  // artifact slot - no online spans, or every query in its request's final
  // span -, keys read from the pool, every slot read, 2 or more requests'
  // rows per CTA)
  int32_t opt_share = 0;
  int32_t k_by_slot = 0;      // keys rotated at assembly: reads cannot be shared
};

// The slots [lo, hi) of a request that a launch reads, out of its nab artifact
// slots and nsuf chunks of online rows (kv_part as in SplitPolicy).
ATT_HD void kv_part_range(int kv_part, int nab, int nsuf, int& lo, int& hi) {
  lo = (kv_part == 2) ? nab : 0;
  hi = (kv_part == 1) ? nab : nab + nsuf;
}

// Split-KV decomposition of one attention launch over S query rows and S_kv
// online rows per request (tc: the tcgen05 kernel, else the warp-MMA kernel).
// Fails (INVALID_ARG, `err` set) only where the launch would need 2^31 or more CTAs.
attuner_status split_work(const SplitPolicy& pol, const PlanTables& t, int S, int S_kv, bool tc, WorkTable& w,
                          std::string& err);

}  // namespace att
