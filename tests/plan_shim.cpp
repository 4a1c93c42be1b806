// plan_shim.cpp - C entry points over the library's host-only planning code
// (csrc/plan.cpp), compiled with the host compiler alone so that the CPU tests
// can drive request assembly and the split-KV decomposition without a GPU.
#include <string.h>

#include <algorithm>
#include <string>
#include <vector>

#include "plan.h"

static std::string g_err;

extern "C" const char* shim_last_error(void) { return g_err.c_str(); }

// Registry of n_arts artifacts (first block, length); writes into out (capacity
// cap int32 values) the tables of the plan, concatenated:
//   blk_off[n_req+1] | blocks | t_art[n_req] | o_rows[n_req] | span_off[n_req+1]
//   | spans | req_art_off[n_req+1] | art_ids
// and lens[0..3] = sizes of blocks, spans, art_ids and max_o_rows.
extern "C" int shim_assemble(const int32_t* first, const int32_t* L, int32_t n_arts, const int32_t* items,
                             const int32_t* offs, int32_t n_req, int32_t layout, int32_t* out, int64_t cap,
                             int64_t* lens) {
  std::vector<att::Artifact> arts;
  for (int i = 0; i < n_arts; ++i)
    arts.push_back(att::Artifact{first[i], L[i], (L[i] + att::kBlockTokens - 1) / att::kBlockTokens});
  att::PlanTables t;
  const attuner_status s = att::build_plan_tables(arts, items, offs, n_req, layout != 0, t, g_err);
  if (s != ATTUNER_OK) return s;
  std::vector<int32_t> h;
  for (const auto* v : {&t.blk_off, &t.blocks, &t.t_art, &t.o_rows, &t.span_off, &t.spans, &t.req_art_off,
                        &t.art_ids})
    h.insert(h.end(), v->begin(), v->end());
  if ((int64_t)h.size() > cap) {
    g_err = "output capacity too small";
    return ATTUNER_ERR_INVALID_ARG;
  }
  memcpy(out, h.data(), h.size() * sizeof(int32_t));
  lens[0] = (int64_t)t.blocks.size();
  lens[1] = (int64_t)t.spans.size();
  lens[2] = (int64_t)t.art_ids.size();
  lens[3] = t.max_o_rows;
  return ATTUNER_OK;
}

// The plan of shim_assemble's arguments, exported as attuner_plan_export does.
extern "C" int shim_export(const int32_t* first, const int32_t* L, int32_t n_arts, const int32_t* items,
                           const int32_t* offs, int32_t n_req, int32_t layout, int32_t* block_table,
                           int32_t* valid_len, int32_t* index_map, int32_t* token_art, int32_t* token_off,
                           int64_t* sizes) {
  std::vector<att::Artifact> arts;
  for (int i = 0; i < n_arts; ++i)
    arts.push_back(att::Artifact{first[i], L[i], (L[i] + att::kBlockTokens - 1) / att::kBlockTokens});
  att::PlanTables t;
  const attuner_status s = att::build_plan_tables(arts, items, offs, n_req, layout != 0, t, g_err);
  if (s != ATTUNER_OK) return s;
  return att::export_plan_tables(t, block_table, valid_len, index_map, token_art, token_off, sizes, g_err);
}

// Split-KV decomposition of a launch over a plan given by its blk_off and
// o_rows; out = n_req, row_tiles, chunk_blocks, n_cta, cluster, base[n_req],
// nsplit[n_req].  pol = n_q_heads, n_kv_heads, num_sms, opt_split, opt_merge,
// tc_clusters[9].
extern "C" int shim_split_part(const int32_t* pol, const int32_t* blk_off, const int32_t* o_rows, int32_t n_req,
                               int32_t S, int32_t S_kv, int32_t tc, int32_t kv_part, int32_t* out);

extern "C" int shim_split(const int32_t* pol, const int32_t* blk_off, const int32_t* o_rows, int32_t n_req,
                          int32_t S, int32_t S_kv, int32_t tc, int32_t* out) {
  return shim_split_part(pol, blk_off, o_rows, n_req, S, S_kv, tc, 0, out);
}

// As shim_split, for a launch that reads only some slots of each request:
// kv_part 1 the plan's artifact slots, 2 the chunks of the online rows.
extern "C" int shim_split_part(const int32_t* pol, const int32_t* blk_off, const int32_t* o_rows, int32_t n_req,
                               int32_t S, int32_t S_kv, int32_t tc, int32_t kv_part, int32_t* out) {
  if (n_req < 1 || n_req > att::kMaxReq) return ATTUNER_ERR_INVALID_ARG;
  att::SplitPolicy p;
  p.kv_part = kv_part;
  p.n_q_heads = pol[0];
  p.n_kv_heads = pol[1];
  p.num_sms = pol[2];
  p.opt_split = pol[3];
  p.opt_merge = pol[4];
  for (int i = 0; i < 9; ++i) p.tc_clusters[i] = pol[5 + i];
  att::PlanTables t;
  t.n_req = n_req;
  t.blk_off.assign(blk_off, blk_off + n_req + 1);
  t.o_rows.assign(o_rows, o_rows + n_req);
  att::WorkTable w;
  const attuner_status s = att::split_work(p, t, S, S_kv, tc != 0, w, g_err);
  if (s != ATTUNER_OK) return s;
  out[0] = w.n_req;
  out[1] = w.row_tiles;
  out[2] = w.chunk_blocks;
  out[3] = w.n_cta;
  out[4] = w.cluster;
  for (int r = 0; r < n_req; ++r) {
    out[5 + r] = w.base[r];
    out[5 + n_req + r] = w.nsplit[r];
  }
  return ATTUNER_OK;
}

// The Q projection's launch shape: pol = head_dim, hidden, num_sms, opt_rows,
// opt_split; out = {mr, ks} ({0, 0}: no supported shape).
extern "C" void shim_qproj_shape(const int32_t* pol, int32_t heads, int32_t M, int32_t n_lora, int32_t* out) {
  att::QpPolicy p;
  p.head_dim = pol[0];
  p.hidden = pol[1];
  p.num_sms = pol[2];
  p.opt_rows = pol[3];
  p.opt_split = pol[4];
  const att::QpShape s = att::choose_qproj_shape(p, heads, M, n_lora);
  out[0] = s.mr;
  out[1] = s.ks;
}

extern "C" int shim_qproj_supported(int32_t D, int32_t mr, int32_t ks, int32_t n_lora) {
  return att::qproj_shape_supported(D, mr, ks, n_lora) ? 1 : 0;
}

// Shared reads: the plan of (first, L, items, offs) and the split-KV work of
// one warp-MMA launch over it.  pol = n_q_heads, n_kv_heads, num_sms,
// opt_split, opt_share, k_by_slot, kv_part, layout (items < 0: online spans).  out (capacity cap) = n_cta,
// chunk_blocks, share, members, n_dist, art_units, suf_chunks, n_part,
// whole_refs, base[n_req] | nsplit[n_dist + 1] | ref_req | ref_slot |
// ref_nblk | dist_off[n_dist + 1] | dist_refs | dist_src | dist_nb |
// dref_req | dref_j | dref_nref; lens = n_refs, n_dist.
extern "C" int shim_share(const int32_t* pol, const int32_t* first, const int32_t* L, int32_t n_arts,
                          const int32_t* items, const int32_t* offs, int32_t n_req, int32_t S, int32_t S_kv,
                          int32_t* out, int64_t cap, int64_t* lens) {
  std::vector<att::Artifact> arts;
  for (int i = 0; i < n_arts; ++i)
    arts.push_back(att::Artifact{first[i], L[i], (L[i] + att::kBlockTokens - 1) / att::kBlockTokens});
  att::PlanTables t;
  attuner_status s = att::build_plan_tables(arts, items, offs, n_req, pol[7] != 0, t, g_err);
  if (s != ATTUNER_OK) return s;
  att::SplitPolicy p;
  p.n_q_heads = pol[0];
  p.n_kv_heads = pol[1];
  p.num_sms = pol[2];
  p.opt_split = pol[3];
  p.opt_merge = 0;
  p.opt_share = pol[4];
  p.k_by_slot = pol[5];
  p.kv_part = pol[6];
  for (int i = 0; i < 9; ++i) p.tc_clusters[i] = 0;
  att::WorkTable w;
  s = att::split_work(p, t, S, S_kv, false, w, g_err);
  if (s != ATTUNER_OK) return s;
  std::vector<int32_t> h = {w.n_cta,     w.chunk_blocks, w.share,  w.members,   w.n_dist,
                            w.art_units, w.suf_chunks,   w.n_part, w.whole_refs};
  h.insert(h.end(), w.base, w.base + n_req);
  if (w.share) h.insert(h.end(), w.nsplit, w.nsplit + w.n_dist + 1);
  for (const auto* v : {&t.ref_req, &t.ref_slot, &t.ref_nblk, &t.dist_off, &t.dist_refs, &t.dist_src, &t.dist_nb,
                        &t.dref_req, &t.dref_j, &t.dref_nref})
    h.insert(h.end(), v->begin(), v->end());
  if ((int64_t)h.size() > cap) {
    g_err = "output capacity too small";
    return ATTUNER_ERR_INVALID_ARG;
  }
  memcpy(out, h.data(), h.size() * sizeof(int32_t));
  lens[0] = (int64_t)t.ref_req.size();
  lens[1] = t.n_dist();
  return ATTUNER_OK;
}
