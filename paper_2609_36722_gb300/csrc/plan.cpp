// plan.cpp - host-only planning (see plan.h): request assembly into a block
// table (the runtime-order concatenation of independently stored artifact
// caches, Sec. 2.1) and the split-KV decomposition of an attention launch.
#include "plan.h"

#include <algorithm>

namespace att {

namespace {
attuner_status bad(attuner_status s, std::string& err, const std::string& msg) {
  err = msg;
  return s;
}
}  // namespace

attuner_status build_plan_tables(const std::vector<Artifact>& arts, const int32_t* items, const int32_t* offs,
                                 int32_t n_req, bool layout, PlanTables& t, std::string& err) {
  if (n_req < 1 || n_req > kMaxReq)
    return bad(ATTUNER_ERR_INVALID_ARG, err, "n_req must be in [1, " + std::to_string(kMaxReq) + "]");
  if (offs == nullptr) return bad(ATTUNER_ERR_INVALID_ARG, err, "req_offsets_host must not be NULL");
  if (offs[0] != 0) return bad(ATTUNER_ERR_INVALID_ARG, err, "req_offsets_host[0] must be 0");
  for (int i = 0; i < n_req; ++i)
    if (offs[i + 1] < offs[i]) return bad(ATTUNER_ERR_INVALID_ARG, err, "req_offsets_host must be non-decreasing");
  if (offs[n_req] != 0 && items == nullptr)
    return bad(ATTUNER_ERR_INVALID_ARG, err, "artifact_ids_host must not be NULL");
  t = PlanTables();
  {
    // sizes first: the tables grow once
    size_t nblk = 0, nids = 0;
    for (int i = 0; i < offs[n_req]; ++i) {
      const long long a = items[i];
      if (a >= 0 && a < (long long)arts.size()) {
        nblk += arts[a].n_blocks;
        ++nids;
      }
    }
    t.blocks.reserve(nblk);
    t.art_ids.reserve(nids);
    t.art_used.reserve(nids);
  }
  t.n_req = n_req;
  t.req_off.assign(offs, offs + n_req + 1);
  t.blk_off.push_back(0);
  t.span_off.push_back(0);
  for (int r = 0; r < n_req; ++r) {
    long long tok = 0, o = 0;
    const int32_t first_slot = (int32_t)t.blocks.size();
    for (int i = offs[r]; i < offs[r + 1]; ++i) {
      const int a = items[i];
      if (a < 0 && layout) {
        // an online span takes no slot: its rows are online rows o .. o + n - 1,
        // read with every other online row after the artifact slots
        const long long n = -(long long)a;
        t.spans.insert(t.spans.end(), {(int32_t)o, (int32_t)n, (int32_t)t.blocks.size() - first_slot, (int32_t)tok});
        o += n;
        if (o >= (1 << 22)) return bad(ATTUNER_ERR_INVALID_ARG, err, "online rows of a request must be < 2^22");
        continue;
      }
      if (a < 0 || a >= (int)arts.size())
        return bad(ATTUNER_ERR_UNKNOWN_ARTIFACT, err, "artifact id " + std::to_string(a) + " was never registered");
      t.art_ids.push_back(a);
      const Artifact& A = arts[a];
      t.art_used.push_back(A);
      for (int b = 0; b < A.n_blocks; ++b)
        t.blocks.push_back(((A.first_block + b) << 7) | std::min(kBlockTokens, A.L - kBlockTokens * b));
      tok += A.L;
    }
    if (tok + o >= (1ll << 30))
      return bad(ATTUNER_ERR_INVALID_ARG, err, "assembled length of a request must be < 2^30 tokens");
    if (t.blocks.size() >= (size_t)1 << 30)
      return bad(ATTUNER_ERR_INVALID_ARG, err, "a plan must hold < 2^30 blocks in all");
    t.blk_off.push_back((int32_t)t.blocks.size());
    t.t_art.push_back((int32_t)tok);
    t.o_rows.push_back((int32_t)o);
    t.span_off.push_back((int32_t)(t.spans.size() / 4));
    t.max_o_rows = std::max(t.max_o_rows, (int32_t)o);
  }
  t.req_art_off.push_back(0);
  int k = 0;
  for (int r = 0; r < n_req; ++r) {
    for (int i = offs[r]; i < offs[r + 1]; ++i) k += items[i] >= 0;
    t.req_art_off.push_back(k);
  }
  const int n_refs = (int)t.art_ids.size();
  t.ref_req.resize(n_refs);
  t.ref_slot.resize(n_refs);
  t.ref_nblk.resize(n_refs);
  for (int r = 0; r < n_req; ++r) {
    int slot = 0;
    for (int i = t.req_art_off[r]; i < t.req_art_off[r + 1]; ++i) {
      t.ref_req[i] = r;
      t.ref_slot[i] = slot;
      t.ref_nblk[i] = t.art_used[i].n_blocks;
      slot += t.art_used[i].n_blocks;
    }
  }
  t.dist_refs.resize(n_refs);
  for (int i = 0; i < n_refs; ++i) t.dist_refs[i] = i;
  std::stable_sort(t.dist_refs.begin(), t.dist_refs.end(),
                   [&](int32_t x, int32_t y) { return t.art_ids[x] < t.art_ids[y]; });
  t.dist_off.push_back(0);
  for (int i = 1; i < n_refs; ++i)
    if (t.art_ids[t.dist_refs[i]] != t.art_ids[t.dist_refs[i - 1]]) t.dist_off.push_back(i);
  if (n_refs > 0) t.dist_off.push_back(n_refs);
  const int nd = t.n_dist();
  t.dist_src.resize(nd);
  t.dist_nb.resize(nd);
  for (int d = 0; d < nd; ++d) {
    const int i0 = t.dist_refs[t.dist_off[d]];
    t.dist_src[d] = t.blk_off[t.ref_req[i0]] + t.ref_slot[i0];
    t.dist_nb[d] = t.ref_nblk[i0];
  }
  t.dref_req.resize(n_refs);
  t.dref_j.resize(n_refs);
  t.dref_nref.resize(n_refs);
  for (int k = 0; k < n_refs; ++k) {
    const int i = t.dist_refs[k], r = t.ref_req[i];
    t.dref_req[k] = r;
    t.dref_j[k] = i - t.req_art_off[r];
    t.dref_nref[k] = t.req_art_off[r + 1] - t.req_art_off[r];
  }
  return ATTUNER_OK;
}

attuner_status export_plan_tables(const PlanTables& t, int32_t* block_table, int32_t* valid_len,
                                  int32_t* index_map, int32_t* token_art, int32_t* token_off, int64_t* sizes,
                                  std::string& err) {
  if (sizes == nullptr) return bad(ATTUNER_ERR_INVALID_ARG, err, "plan and sizes_inout must not be NULL");
  int64_t nb = 0;
  for (int32_t e : t.blocks) nb += e > 0;   // artifact blocks (online chunks are not exported)
  int64_t nt = 0;
  for (int32_t v : t.t_art) nt += v;
  if (block_table && sizes[0] < nb) return bad(ATTUNER_ERR_INVALID_ARG, err, "block_table capacity too small");
  if (valid_len && sizes[1] < nb) return bad(ATTUNER_ERR_INVALID_ARG, err, "valid_len capacity too small");
  if (index_map && sizes[2] < nt) return bad(ATTUNER_ERR_INVALID_ARG, err, "index_map capacity too small");
  if (token_art && sizes[3] < nt) return bad(ATTUNER_ERR_INVALID_ARG, err, "token_art capacity too small");
  if (token_off && sizes[4] < nt) return bad(ATTUNER_ERR_INVALID_ARG, err, "token_off capacity too small");
  {
    int64_t i = 0;
    for (int32_t e : t.blocks) {
      if (e <= 0) continue;
      if (block_table) block_table[i] = e >> 7;
      if (valid_len) valid_len[i] = e & 127;
      ++i;
    }
  }
  int64_t tok = 0;
  for (int r = 0; r < t.n_req; ++r) {
    for (int i = t.req_art_off[r]; i < t.req_art_off[r + 1]; ++i) {
      const int a = t.art_ids[i];
      const Artifact& A = t.art_used[i];
      for (int q = 0; q < A.L; ++q, ++tok) {
        if (index_map) index_map[tok] = (A.first_block + q / kBlockTokens) * kBlockTokens + q % kBlockTokens;
        if (token_art) token_art[tok] = a;
        if (token_off) token_off[tok] = q;
      }
    }
  }
  sizes[0] = nb;
  sizes[1] = nb;
  sizes[2] = nt;
  sizes[3] = nt;
  sizes[4] = nt;
  sizes[5] = t.n_req;
  return ATTUNER_OK;
}

namespace {
constexpr long long kMaxCta = 0x7fffffffll;

// The shared-read decomposition (see WorkTable); reads_share = block reads of
// the artifact units per KV head.
attuner_status share_work(const SplitPolicy& pol, const PlanTables& t, int S_kv, int members, long long reads_share,
                          WorkTable& w, std::string& err) {
  const int Hkv = pol.n_kv_heads, nd = t.n_dist();
  const int nsuf = (S_kv + kBlockTokens - 1) / kBlockTokens;
  int chunk = pol.opt_split;
  if (chunk <= 0) {
    // The groups already give many CTAs, and every further chunk of an
    // artifact adds a partial result to each of its requests: about eight
    // CTAs per SM, at least 32 blocks (on the 64-request decode step, whose
    // artifacts have 4 to 32 blocks, chunks of 12, 16, 24, 32 and 64 blocks
    // took 0.253, 0.232, 0.224, 0.212 and 0.212 ms).
    const long long total = (reads_share + (long long)t.n_req * nsuf) * Hkv;
    const long long target = 8ll * pol.num_sms;
    chunk = (int)std::max<long long>(32, (total + target - 1) / target);
  }
  chunk = std::min(chunk, kMmaMaxChunkBlocks);
  auto nch = [&](long long nb) { return (nb + chunk - 1) / chunk; };
  w.n_req = t.n_req;
  w.row_tiles = 1;
  w.chunk_blocks = chunk;
  w.cluster = 0;
  w.share = 1;
  w.members = members;
  w.n_dist = nd;
  w.whole_refs = 1;
  for (int32_t nb : t.dist_nb) w.whole_refs &= (nb <= chunk) ? 1 : 0;
  long long u = 0;
  for (int d = 0; d < nd; ++d) {
    w.nsplit[d] = (int32_t)u;
    const int nref = t.dist_off[d + 1] - t.dist_off[d];
    u += nch(t.dist_nb[d]) * ((nref + members - 1) / members);
    if (u * Hkv > kMaxCta) return bad(ATTUNER_ERR_INVALID_ARG, err, "attention launch needs >= 2^31 CTAs");
  }
  w.nsplit[nd] = (int32_t)u;
  w.art_units = (int32_t)u;
  w.suf_chunks = (int32_t)nch(nsuf);
  const long long per_head = u + (long long)t.n_req * w.suf_chunks;
  if (per_head * Hkv > kMaxCta) return bad(ATTUNER_ERR_INVALID_ARG, err, "attention launch needs >= 2^31 CTAs");
  long long part = 0;
  for (int r = 0; r < t.n_req; ++r) {
    w.base[r] = (int32_t)part;
    for (int i = t.req_art_off[r]; i < t.req_art_off[r + 1]; ++i) part += nch(t.ref_nblk[i]);
    part += w.suf_chunks;
  }
  if (part * Hkv > kMaxCta) return bad(ATTUNER_ERR_INVALID_ARG, err, "attention launch needs >= 2^31 partials");
  w.n_part = (int32_t)part;
  w.n_cta = (int32_t)(per_head * Hkv);
  return ATTUNER_OK;
}
}  // namespace

attuner_status split_work(const SplitPolicy& pol, const PlanTables& t, int S, int S_kv, bool tc, WorkTable& w,
                          std::string& err) {
  w.share = 0;
  w.members = 0;
  w.n_dist = 0;
  w.art_units = 0;
  w.suf_chunks = 0;
  w.n_part = 0;
  w.whole_refs = 0;
  const int G = pol.n_q_heads / pol.n_kv_heads, Hkv = pol.n_kv_heads;
  const int rows = tc ? kTcRows : kMmaRows;
  const int row_tiles = (S * G + rows - 1) / rows;
  // slots of request r the launch reads: the plan's artifact slots, then the
  // 64-row chunks of its online rows (or one of the two, kv_part)
  auto nslots = [&](int r) {
    int lo, hi;
    kv_part_range(pol.kv_part, t.blk_off[r + 1] - t.blk_off[r], (S_kv + kBlockTokens - 1) / kBlockTokens, lo, hi);
    return hi - lo;
  };
  long long total = 0;
  int maxv = 0;
  for (int r = 0; r < t.n_req; ++r) {
    const int nv = nslots(r);
    total += (long long)nv * Hkv * row_tiles;
    maxv = std::max(maxv, nv);
  }
  const long long units = (long long)t.n_req * Hkv * row_tiles;
  w.n_req = t.n_req;
  w.row_tiles = row_tiles;
  if (maxv == 0) {   // no request has a slot to read (a part-only launch): no CTA
    w.cluster = 0;
    w.chunk_blocks = tc ? 2 : 16;
    for (int r = 0; r < t.n_req; ++r) {
      w.base[r] = 0;
      w.nsplit[r] = 0;
    }
    w.n_cta = 0;
    return ATTUNER_OK;
  }
  // Shared reads (warp-MMA kernel): a CTA reads a chunk of one artifact for up
  // to `members` requests that use it.  Taken where it saves 10 % or more of
  // the block reads (or always, opt_share = 2, where it applies).  Every query
  // must see every artifact slot: in a prompt layout, every query row sits in
  // its request's final online span (as a decode token does).
  {
    const int SG = S * G;
    const int members = SG <= kMmaRows ? kMmaRows / SG : 0;
    const int nd = t.n_dist();
    bool all_see_all = true;
    for (int r = 0; r < t.n_req && t.max_o_rows > 0; ++r) all_see_all &= S <= S_kv - t.o_rows[r];
    if (!tc && pol.opt_share != 1 && members >= 2 && pol.kv_part == 0 && all_see_all && !pol.k_by_slot &&
        nd > 0 && nd <= kMaxShareArts) {
      long long reads_req = 0, reads_share = 0;
      for (int d = 0; d < nd; ++d) {
        const int nref = t.dist_off[d + 1] - t.dist_off[d];
        const long long nb = t.dist_nb[d];
        reads_req += nb * nref;
        reads_share += nb * ((nref + members - 1) / members);
      }
      if (pol.opt_share == 2 || reads_share * 10 <= reads_req * 9)
        return share_work(pol, t, S_kv, members, reads_share, w, err);
    }
  }
  // Cluster mode (tcgen05 kernel): every row tile cut into ns (2 or 4)
  // chunks, one cluster of ns CTAs per row tile.  Cost in 128-key tile times: waves of
  // co-resident clusters x (largest chunk + ~4 tiles of prologue and epilogue
  // + ~1 for the merge).
  auto cluster_cost = [&](int ns) -> double {
    const int maxc = pol.tc_clusters[ns];
    if (maxc <= 0) return 1e30;
    const int chunk = (((maxv + ns - 1) / ns) + 1) & ~1;
    if (chunk > kMaxChunkBlocks) return 1e30;
    const long long waves = (units + maxc - 1) / maxc;
    return (double)waves * (chunk / 2 + 5.0);
  };
  int cluster_ns = 0;
  int chunk;
  if (pol.opt_split > 0) {
    chunk = pol.opt_split;
    // a cluster merges 2 or 4 chunks (whole column blocks per CTA); where such
    // clusters cannot be co-resident the chunks merge through global memory
    if (tc && pol.opt_merge == 2 && maxv > chunk) {
      cluster_ns = (maxv + chunk - 1) / chunk <= 2 ? 2 : 4;
      if ((((maxv + cluster_ns - 1) / cluster_ns) + 1) / 2 * 2 > kMaxChunkBlocks || pol.tc_clusters[cluster_ns] <= 0)
        cluster_ns = 0;
    }
  } else if (tc) {
    // Independent splits, one CTA per SM.  Cost of a chunk size = waves x
    // (tiles per CTA + ~4 tiles for the prologue and epilogue + ~2 for the
    // merge through global memory + ~0.35 per further split, the time the
    // merging CTA spends reading one more 17 KiB-per-32-column partial back);
    // pick the number of splits of the longest request that minimises it.
    // (On the 131k-key layer 4 and 7 splits take the same time; the read-back
    // term picks 4, which writes and reads half the partial bytes.  Plans with
    // online spans leave it out: their row tiles read different numbers of
    // artifact slots, and finer chunks balance them - the 131k-key skills
    // layout took 2.93 ms with 7 chunks per row tile, 3.04 ms with 4.)
    const int maxt = (maxv + 1) / 2;
    double best = 1e30;
    chunk = maxv;
    if (pol.opt_merge != 2) {
      for (int sp = 1; sp <= kMaxSplits; ++sp) {
        const int ct = (maxt + sp - 1) / sp;
        long long ncta = 0;
        for (int r = 0; r < t.n_req; ++r) {
          const int nv = nslots(r);
          ncta += (long long)((nv + 2 * ct - 1) / (2 * ct)) * Hkv * row_tiles;
        }
        const long long waves = (ncta + pol.num_sms - 1) / pol.num_sms;
        const double readback = t.max_o_rows > 0 ? 0.0 : 0.35 * (sp - 1);
        const double cost = (double)waves * (ct + 4.0 + (sp > 1 ? 2.0 + readback : 0.0));
        if (cost < best - 1e-9) {
          best = cost;
          chunk = 2 * ct;
        }
      }
    }
    if (pol.opt_merge != 1) {
      for (int ns = 2; ns <= 4; ns += 2) {   // a cluster merges 2 or 4 chunks
        const double cost = cluster_cost(ns);
        if (cost < best - 1e-9) {
          best = cost;
          cluster_ns = ns;
        }
      }
    }
  } else {
    // decode: about sixteen small CTAs per SM, two resident at a time (on
    // the 64-request decode step chunks of 24, 32, 48 and 65 blocks took
    // 0.298, 0.290, 0.296 and 0.311 ms), balancing requests of different lengths
    const long long target = 16ll * pol.num_sms;
    chunk = (int)std::max<long long>(16, (total + target - 1) / target);
  }
  w.n_req = t.n_req;
  w.row_tiles = row_tiles;
  if (cluster_ns > 0) {
    w.cluster = cluster_ns;
    w.chunk_blocks = 0;   // per request, ceil(blocks / cluster) rounded up to whole tiles
    for (int r = 0; r < t.n_req; ++r) {
      w.base[r] = (int)(r * (long long)Hkv * row_tiles * cluster_ns);
      w.nsplit[r] = cluster_ns;
    }
    if (units * cluster_ns > kMaxCta) return bad(ATTUNER_ERR_INVALID_ARG, err, "attention launch needs >= 2^31 CTAs");
    w.n_cta = (int)(units * cluster_ns);
    return ATTUNER_OK;
  }
  w.cluster = 0;
  chunk = std::min(chunk, tc ? kMaxChunkBlocks : kMmaMaxChunkBlocks);
  if (tc) {
    // the kernel merges at most kMaxSplits chunks of one row tile
    chunk = std::max(chunk, (maxv + kMaxSplits - 1) / kMaxSplits);
    chunk = (chunk + 1) & ~1;   // whole 128-key tiles per split
  }
  w.chunk_blocks = chunk;
  long long base = 0;
  for (int r = 0; r < t.n_req; ++r) {
    const int nv = nslots(r);
    const int ns = (nv + chunk - 1) / chunk;
    w.base[r] = (int32_t)base;
    w.nsplit[r] = ns;
    base += (long long)ns * Hkv * row_tiles;
    if (base > kMaxCta)
      return bad(ATTUNER_ERR_INVALID_ARG, err, "attention launch needs >= 2^31 CTAs (use larger split chunks)");
  }
  w.n_cta = (int32_t)base;
  return ATTUNER_OK;
}

bool qproj_shape_supported(int D, int mr, int ks, int n_lora) {
  if (D != 64 && D != 128) return false;
  if (mr != 1 && mr != 2) return false;
  if (ks != 1 && ks != 2 && ks != 4 && ks != 8) return false;
  if (ks == 1) return true;
  const int tpr = ks / mr;
  if (tpr < 1 || D / 2 / tpr < 8) return false;
  return qp_recv_bytes(mr, D, qp_lora_width(n_lora)) <= qp_ring_bytes(D, mr);
}

// The estimate is waves x (start-up + operand bytes + epilogue), with
// constants from per-CTA timelines on GB300: about 2.5 us from launch to the
// first full stage; the operand stream, (mr*128 + D + r) * hidden/ks * 2 bytes
// per CTA (out-of-range rows of a tile are filled, not skipped), at about
// 100 GB/s per SM; an epilogue of about 3.5 us, plus 1.5 us and the exchanged
// partial rows at about 20 GB/s when the K dimension is split.
QpShape choose_qproj_shape(const QpPolicy& pol, int heads, int M, int n_lora) {
  const int D = pol.head_dim, nk = pol.hidden / 64;
  QpShape best{0, 0};
  double best_t = 0.0;
  for (int mr = 1; mr <= 2; ++mr)
    for (int ks = 1; ks <= 8; ks *= 2) {
      if (pol.opt_rows != 0 && pol.opt_rows != 128 * mr) continue;
      if (pol.opt_split != 0 && pol.opt_split != ks) continue;
      if (ks > nk || !qproj_shape_supported(D, mr, ks, n_lora)) continue;
      const long long tiles = (long long)heads * ((M + 128 * mr - 1) / (128 * mr));
      const long long waves = (tiles * ks + pol.num_sms - 1) / pol.num_sms;
      const double bytes = (double)(128 * mr + D + n_lora) * (double)(pol.hidden / ks) * 2.0;
      const double exch = (double)std::min(128 * mr, M) * (D + n_lora) * 4.0;
      const double epi = ks > 1 ? 5.0e-6 + exch / 20e9 : 3.5e-6;
      const double t = (double)waves * (2.5e-6 + bytes / 100e9 + epi);
      if (best.mr == 0 || t < best_t) {
        best = {mr, ks};
        best_t = t;
      }
    }
  return best;
}

}  // namespace att
