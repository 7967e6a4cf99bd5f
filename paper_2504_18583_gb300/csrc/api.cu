// C ABI of libpard: context set-up and the launch sequences of the PARD
// decode step (prefill, draft, verify, accept/commit).
//
// The library never allocates device memory: the caller's workspace is
// carved into activation buffers, reduction scratch, row plans and the
// per-sequence state; the caller's page pool holds both models' KV caches.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <set>
#include <string>
#include <vector>

#include "common.cuh"
#include "internal.h"

using namespace pard;

namespace {

thread_local std::string g_err;

pard_status fail(pard_status st, const std::string& msg) {
  g_err = msg;
  return st;
}

struct CudaFail {
  cudaError_t e;
  const char* what;
};

}  // namespace

// error message shared with the other translation units of the library
namespace pard {
void set_error(const std::string& msg) { g_err = msg; }
}  // namespace pard

namespace {
#define CK(x)                                           \
  do {                                                  \
    cudaError_t e_ = (x);                               \
    if (e_ != cudaSuccess) throw CudaFail{e_, #x};      \
  } while (0)

// ---- model description -----------------------------------------------------
struct LayerW {
  const __nv_bfloat16* t[9];  // attn_norm, wq, wk, wv, wo, mlp_norm, wg, wu, wd
};
enum { W_ATTN_NORM, W_Q, W_K, W_V, W_O, W_MLP_NORM, W_G, W_U, W_D };

struct LayerMaps {
  CUtensorMap q, k, v, o, g, u, dn;
};

struct Model {
  pard_model_cfg cfg;
  const __nv_bfloat16* embed = nullptr;
  const __nv_bfloat16* final_norm = nullptr;
  const __nv_bfloat16* lm_head = nullptr;
  std::vector<LayerW> L;
  std::vector<LayerW> P;        // packed matrices (same pointers) or null where row-major
  std::vector<LayerMaps> maps;
  CUtensorMap lm_map;
  const __nv_bfloat16* lm_pk = nullptr;
  __nv_bfloat16* kv = nullptr;  // [layer][K|V][page][hkv][ps][hd]
  size_t page_elems = 0;        // hkv * ps * hd
  int* page_table = nullptr;    // [max_batch][pt_ld]
  float2* rope = nullptr;       // [max_ctx][hd/2]
  int qd() const { return cfg.n_q_heads * cfg.head_dim; }
  int kvd() const { return cfg.n_kv_heads * cfg.head_dim; }
  __nv_bfloat16* kcache(int l) const { return kv + (size_t)(2 * l) * n_pages_ * page_elems; }
  __nv_bfloat16* vcache(int l) const { return kv + (size_t)(2 * l + 1) * n_pages_ * page_elems; }
  int n_pages_ = 0;
};

// ---- workspace layout ------------------------------------------------------
struct Layout {
  size_t total = 0;
  size_t take(size_t bytes) {
    size_t off = (total + 255) & ~size_t(255);
    total = off + bytes;
    return off;
  }
};

struct Dims {
  int MC;           // row capacity of every row-indexed buffer
  int m_dec;        // rows of a decode pass (B * 2K)
  int gcap;         // rows of the prefill LM-head input
  int dmax, qdmax, ffnmax, vocab, hkvmax, hdmax, w_tiles, pt_ld, sm;
  int ffn_pad;      // widest FFN rounded up to whole 64-column blocks
};

int round_up(int x, int m) { return (x + m - 1) / m * m; }

Dims make_dims(const pard_model_cfg& t, const pard_model_cfg& d, const pard_limits& lim, int sm) {
  Dims D;
  D.m_dec = lim.max_batch * 2 * lim.max_k;
  // whole token tiles of the widest pass (tiles of 128 rows above 64)
  const int mrows = std::max(D.m_dec, lim.prefill_chunk);
  D.MC = round_up(mrows, mrows > 64 ? 128 : 64);
  // whole token tiles of the LM-head input
  D.gcap = lim.max_batch <= 16 ? 16 : (lim.max_batch <= 64 ? 64 : round_up(lim.max_batch, 128));
  D.dmax = std::max(t.d_model, d.d_model);
  D.qdmax = std::max(t.n_q_heads * t.head_dim, d.n_q_heads * d.head_dim);
  D.ffnmax = std::max(t.ffn, d.ffn);
  D.ffn_pad = round_up(D.ffnmax, 64);
  D.vocab = t.vocab;
  D.hkvmax = std::max(t.n_kv_heads, d.n_kv_heads);
  D.hdmax = std::max(t.head_dim, d.head_dim);
  D.w_tiles = (t.vocab + kTileN - 1) / kTileN;
  D.pt_ld = (lim.max_ctx + lim.page_size - 1) / lim.page_size;
  D.sm = sm;
  return D;
}

constexpr size_t kPackTmpBytes = (size_t)32 << 20;  // scratch for in-place weight packing

struct WsOffsets {
  size_t h, xd, xo, xf, xg, ssq, ssqg, q, gpart, gcnt, stats_t, stats_it, stats_d, stats_id, logits, dlogits;
  size_t row_tok, row_pos, row_seq, row_out, row_gi, seq_row0, m_dev;
  size_t g_row_seq, g_row_gi, g_m;
  size_t st_n, st_pc, st_pend, st_gen, st_max, st_done, st_d, st_dnorm, st_sa, st_snorm, st_spart, st_scnt;
  size_t call, status, paths, tmp_pos, pt[2], rope[2], g_plen, pack_tmp, mask_ids;
  size_t total;
};

WsOffsets layout_ws(const Dims& D, const pard_limits& lim) {
  Layout L;
  WsOffsets o;
  const int B = lim.max_batch, K = lim.max_k;
  o.h = L.take((size_t)D.MC * D.dmax * 4);
  o.xd = L.take((size_t)2 * D.MC * D.dmax * 2);
  o.xo = L.take((size_t)2 * D.MC * D.qdmax * 2);
  o.xf = L.take((size_t)2 * D.MC * D.ffn_pad * 2);
  o.xg = L.take((size_t)2 * D.gcap * D.dmax * 2);
  o.ssq = L.take((size_t)(D.dmax / 128) * D.MC * 4);
  o.ssqg = L.take((size_t)(D.dmax / 128) * D.MC * 4);
  o.q = L.take((size_t)D.MC * D.qdmax * 4);
  o.gcnt = L.take((size_t)kMaxGemmTiles * 8);  // one 64-bit arrival mask per output tile
  o.stats_t = L.take((size_t)D.w_tiles * D.MC * 16);
  o.stats_it = L.take((size_t)D.w_tiles * D.MC * 8);
  o.stats_d = L.take((size_t)D.w_tiles * D.MC * 16);
  o.stats_id = L.take((size_t)D.w_tiles * D.MC * 8);
  o.logits = L.take((size_t)B * (K + 1) * D.vocab * 4);
  o.dlogits = L.take((size_t)B * K * D.vocab * 4);
  o.row_tok = L.take((size_t)D.MC * 4);
  o.row_pos = L.take((size_t)D.MC * 4);
  o.row_seq = L.take((size_t)D.MC * 4);
  o.row_out = L.take((size_t)D.MC * 4);
  o.row_gi = L.take((size_t)D.MC * 4);
  o.seq_row0 = L.take((size_t)(B + 1) * 4);
  o.m_dev = L.take(4);
  o.g_row_seq = L.take((size_t)D.gcap * 4);
  o.g_row_gi = L.take((size_t)D.gcap * 4);
  o.g_m = L.take(4);
  o.st_n = L.take((size_t)B * 4);
  o.st_pc = L.take((size_t)B * 4);
  o.st_pend = L.take((size_t)B * (K + 1) * 4);
  o.st_gen = L.take((size_t)B * 4);
  o.st_max = L.take((size_t)B * 4);
  o.st_done = L.take((size_t)B * 4);
  o.st_d = L.take((size_t)B * K * 4);
  o.st_dnorm = L.take((size_t)B * K * 8);
  o.st_sa = L.take((size_t)B * 4);
  o.st_snorm = L.take((size_t)B * 16);
  o.st_spart = L.take((size_t)B * kResampleSplit * 8);
  o.st_scnt = L.take((size_t)B * 4);
  o.call = L.take(sizeof(CallArgs));
  o.status = L.take(4);
  o.paths = L.take(4);
  o.tmp_pos = L.take(4096 * 4);
  for (int mi = 0; mi < 2; ++mi) o.pt[mi] = L.take((size_t)B * D.pt_ld * 4);
  for (int mi = 0; mi < 2; ++mi) o.rope[mi] = L.take((size_t)D.pt_ld * lim.page_size * (D.hdmax / 2) * 8);
  o.g_plen = L.take((size_t)B * 4);
  o.mask_ids = L.take((size_t)std::max(K, 1) * 4);
  o.gpart = L.take((size_t)D.sm * 2 * kTileN * (D.MC > 64 ? 128 : 64) * 4);  // two partial tiles per CTA
  o.pack_tmp = L.take(kPackTmpBytes);
  o.total = L.total + 256;
  return o;
}

bool valid_cfg(const pard_model_cfg* c, std::string& why) {
  if (!c) { why = "null model config"; return false; }
  if (c->n_layers < 1) { why = "n_layers < 1"; return false; }
  if (c->head_dim != 64 && c->head_dim != 128) { why = "head_dim must be 64 or 128"; return false; }
  if (c->n_kv_heads < 1 || c->n_q_heads % c->n_kv_heads) { why = "n_q_heads must be a multiple of n_kv_heads"; return false; }
  const int g = c->n_q_heads / c->n_kv_heads;
  if (g != 1 && g != 2 && g != 4 && g != 8) { why = "GQA group must be 1, 2, 4 or 8"; return false; }
  if (c->d_model % 128 || (c->n_q_heads * c->head_dim) % 128 || (c->n_kv_heads * c->head_dim) % 128) {
    why = "d_model, n_q_heads*head_dim and n_kv_heads*head_dim must be multiples of 128";
    return false;
  }
  if (c->ffn < 8 || c->ffn % 8) { why = "ffn must be a positive multiple of 8"; return false; }
  if (c->vocab < 8 || c->vocab % 8) { why = "vocab must be a positive multiple of 8"; return false; }
  if (c->mask_id < 0 || c->mask_id >= c->vocab) { why = "mask_id outside [0, vocab)"; return false; }
  if (!(c->rope_theta > 0.f) || !(c->rms_eps >= 0.f)) { why = "bad rope_theta or rms_eps"; return false; }
  return true;
}

bool valid_limits(const pard_limits* l, std::string& why) {
  if (!l) { why = "null limits"; return false; }
  if (l->max_batch < 1 || l->max_batch > 64) { why = "max_batch must be in [1, 64]"; return false; }
  if (l->max_k < 1 || l->max_k > 16) { why = "max_k must be in [1, 16]"; return false; }
  if (l->page_size != 16) { why = "page_size must be 16"; return false; }
  if (l->max_ctx < 1 || l->max_ctx > 1 << 20) { why = "bad max_ctx"; return false; }
  if (l->prefill_chunk < 64 || l->prefill_chunk > 1024 || l->prefill_chunk % 64) {
    why = "prefill_chunk must be a multiple of 64 in [64, 1024]";
    return false;
  }
  if (l->n_pages < 1) { why = "n_pages < 1"; return false; }
  return true;
}

size_t kv_bytes_model(const pard_model_cfg& c, const pard_limits& l) {
  return (size_t)c.n_layers * 2 * l.n_pages * c.n_kv_heads * l.page_size * c.head_dim * 2;
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D bf16 row-major [rows][cols] tensor map, box {64 cols, box_rows}, 128B swizzle.
CUtensorMap make_map(const void* base, int rows, int cols, int box_rows) {
  CUtensorMap m;
  std::memset(&m, 0, sizeof(m));
  auto enc = get_encode();
  if (!enc) throw CudaFail{cudaErrorNotSupported, "cuTensorMapEncodeTiled unavailable"};
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {(cuuint32_t)kChunkK, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(&m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) throw CudaFail{cudaErrorInvalidValue, "cuTensorMapEncodeTiled rejected a tensor"};
  return m;
}

// Token tile of a pass of up to `rows` rows: 16, 64, or 128 (65 and more
// rows: one pass over the weights covers 128 of them).
int pick_tt(int rows) { return rows <= 16 ? 16 : (rows <= 64 ? 64 : 128); }

}  // namespace

struct pard_ctx {
  Model m[2];
  pard_limits lim;
  Dims D;
  WsOffsets o;
  uint8_t* ws = nullptr;
  int sm = 0;
  // device views
  float *h, *ssq, *ssqg, *q, *gpart, *logits, *dlogits;
  __nv_bfloat16 *xd, *xo, *xf, *xg;
  int* gcnt;
  float4 *stats_t, *stats_d;
  int2 *stats_it, *stats_id;
  RowPlan rp;
  int *g_row_seq, *g_row_gi, *g_m;
  DevState st;
  CallArgs* call;
  uint32_t* status;
  uint32_t* paths;        // attention combine paths taken since the last read
  int attn_split_cap = kMaxAttnSplit;  // key splits per attention cluster, at most
  int* tmp_pos;
  int* g_plen;
  int* mask_ids;          // per-offset draft mask ids (used when n_mask_ids > 0)
  int n_mask_ids = 0;     // 0: the draft config's shared mask id
  // host state
  std::vector<int> order[2];
  int batch = 0, K = 0, n_new = 0;
  std::vector<int> ctx_est;  // per sequence: prompt + n_new, an upper bound of its context (attention splits)
  bool prefilled = false;
  bool last_draft_sampled = false;
  bool unpacked = false;
  std::vector<std::pair<__nv_bfloat16*, int>> packed_list;  // (matrix, R) packed in place, with N, K below
  std::vector<std::pair<int, int>> packed_shape;
  int launches = 0;
  template <typename T>
  T* at(size_t off) { return reinterpret_cast<T*>(ws + off); }
};

namespace {

void set_call(pard_ctx* c, uint64_t seed, uint64_t step, float temp, int sample, cudaStream_t s) {
  CallArgs v{seed, step, temp, sample, c->K, 0};
  launch_set_call(c->call, v, s, true);
  c->launches++;
}

GemmArgs gemm_base(pard_ctx* c, int rows_cap, int tt) {
  GemmArgs a;
  std::memset(&a, 0, sizeof(a));
  a.tok_tiles = (rows_cap + tt - 1) / tt;
  a.n_tok = a.tok_tiles == 1 ? round_up(rows_cap, 8) : 0;
  a.m_cap = c->D.MC;
  a.m_dev = c->rp.m_dev;
  a.partials = c->gpart;
  a.counters = c->gcnt;
  a.status = c->status;
  a.call = c->call;
  return a;
}

void run_gemm(pard_ctx* c, GemmArgs& a, int tt, cudaStream_t s) {
  const long U = (long)a.w_tiles * a.tok_tiles * a.kc;
  // at least 8 units (128 KB of weights) a CTA: with fewer, the split-K
  // finish of a tile gathers partials from too many CTAs; and at least
  // kc / 62 units, so that no tile has more than 63 contributors (the
  // finisher tracks their arrivals in one 64-bit mask)
  const long min_units = std::max<long>(8, (a.kc + 61) / 62);
  const int grid = (int)std::min<long>(c->sm, std::max<long>(1, U / min_units));
  if ((long)a.w_tiles * a.tok_tiles > kMaxGemmTiles) throw cudaErrorInvalidValue;
  launch_gemm(a, tt, grid, s, true);
  c->launches++;
}

// Attention work decomposition of a pass: row blocks per sequence, groups
// (sequence x kv head x row block) and key splits (<= 16 or the context's
// cap, about two CTAs per SM, at most one per 32-key chunk of the longest
// context).
struct AttnGeom {
  int row_blocks, groups, n_split;
  int nbuf;  // K/V chunk buffers of the attention kernel's form (4, or 2 for passes with many units)
};
AttnGeom attn_geometry(pard_ctx* c, int mi, int rows_per_seq, int batch) {
  const pard_model_cfg& cf = c->m[mi].cfg;
  const int rb_rows = attention_rows_per_block(cf.n_q_heads / cf.n_kv_heads);
  AttnGeom g;
  g.row_blocks = (rows_per_seq + rb_rows - 1) / rb_rows;
  g.groups = batch * cf.n_kv_heads * g.row_blocks;
  const int n_kt = (c->lim.max_ctx + 31) / 32;  // 32-key chunks at the longest context
  g.n_split = std::max(1, std::min({c->attn_split_cap, n_kt, (2 * c->sm + g.groups - 1) / g.groups}));
  g.nbuf = 4;
  long total = 0, longest = 0;
  if (batch > 1 && (int)c->ctx_est.size() >= batch)
    for (int b = 0; b < batch; ++b) {
      const long ch = (c->ctx_est[b] + 31) / 32;
      total += ch;
      longest = std::max(longest, ch);
    }
  const bool ragged = 2 * longest * batch > 3 * total;  // the longest context above 1.5 times the mean
  const bool crowded = (long)g.groups * g.n_split > 2L * c->sm && longest >= 3L * g.n_split;
  if (total > 0 && (ragged || crowded)) {
    // Ragged contexts, where the kernel lasts as long as the longest
    // sequence's units (its chunks / n_split each), or more units than two
    // CTAs per SM that walk three chunks or more: such passes take the
    // two-buffer ring (four CTAs per SM; its warp pairs split the keys of
    // units with three chunks or more) and split until the longest
    // sequence's share is no longer than the average CTA's share of all
    // units' chunks at four CTAs per SM (even contexts: 4 x 152 / groups);
    // more splits only add per-CTA start-up and combine work.  Measured on
    // 512-token contexts: batch 4 (two chunks a unit) is faster with the
    // four-buffer form, batch 8 and 16 with this one.
    total *= (long)cf.n_kv_heads * g.row_blocks;
    const long bal = (longest * 4 * c->sm + total - 1) / total;
    g.n_split = std::max<long>(g.n_split, std::min<long>({bal, (long)c->attn_split_cap, (long)n_kt}));
    g.nbuf = 2;
  }
  return g;
}

// Arguments of the five phases of layer l (QKV, attention, O, gate/up, down).
struct LayerPlan {
  GemmArgs qkv, o, gu, dn;
  AttnArgs at;
};
LayerPlan layer_plan(pard_ctx* c, int mi, int l, int rows_cap, int tt, int tt_gu, int batch, const int* pt_attn,
                     const AttnGeom& geo, int fixed_rows) {
  Model& M = c->m[mi];
  const pard_model_cfg& cf = M.cfg;
  const int d = cf.d_model, qd = M.qd(), kvd = M.kvd(), ffn = cf.ffn;
  const LayerW& W = M.L[l];
  const LayerMaps& Mp = M.maps[l];
  LayerPlan P;
  // fused RMSNorm -> QKV -> RoPE -> paged KV write
  {
    GemmArgs& a = P.qkv;
    a = gemm_base(c, rows_cap, tt);
    a.wmap[0] = Mp.q; a.wmap[1] = Mp.k; a.wmap[2] = Mp.v;
    a.wpk[0] = M.P[l].t[W_Q]; a.wpk[1] = M.P[l].t[W_K]; a.wpk[2] = M.P[l].t[W_V];
    a.x = c->xd; a.x_rows = 2 * c->D.MC;
    a.nseg = 3;
    a.seg_tile0[0] = 0;
    a.seg_tile0[1] = qd / kTileN;
    a.seg_tile0[2] = a.seg_tile0[1] + kvd / kTileN;
    a.seg_tile0[3] = a.seg_tile0[2] + kvd / kTileN;
    a.seg_rows[0] = qd; a.seg_rows[1] = kvd; a.seg_rows[2] = kvd;
    a.w_tiles = a.seg_tile0[3];
    a.kc = (d + kChunkK - 1) / kChunkK;
    a.mode = MODE_QKV;
    a.ssq_in = c->ssq; a.ssq_tiles = d / 128; a.inv_d = 1.0f / d; a.eps = cf.rms_eps;
    a.q_out = c->q; a.q_ld = qd;
    a.kcache = M.kcache(l); a.vcache = M.vcache(l);
    a.page_table = M.page_table; a.pt_ld = c->D.pt_ld;
    a.row_pos = c->rp.row_pos; a.row_seq = c->rp.row_seq;
    a.rope = M.rope; a.hd = cf.head_dim; a.hkv = cf.n_kv_heads; a.page_size = c->lim.page_size;
    a.n_pages = c->lim.n_pages;
  }
  // attention over the paged cache
  {
    AttnArgs& a = P.at;
    std::memset(&a, 0, sizeof(a));
    a.q = c->q; a.q_ld = qd;
    a.kcache = M.kcache(l); a.vcache = M.vcache(l);
    a.page_table = pt_attn; a.pt_ld = c->D.pt_ld;
    a.row_pos = c->rp.row_pos; a.seq_row0 = c->rp.seq_row0; a.rows_per_seq = fixed_rows; a.m_dev = c->rp.m_dev;
    a.batch = batch; a.hq = cf.n_q_heads; a.hkv = cf.n_kv_heads; a.hd = cf.head_dim;
    a.page_size = c->lim.page_size; a.n_pages = c->lim.n_pages;
    a.row_blocks = geo.row_blocks; a.n_split = geo.n_split;
    a.nbuf = geo.nbuf;
    a.scale = (float)(1.0 / std::sqrt((double)cf.head_dim));
    a.x_out = c->xo; a.x_rows = 2 * c->D.MC;
    a.status = c->status;
    a.paths = c->paths;
  }
  // O projection + residual; emits x = h * g_mlp and the new row sums of squares
  {
    GemmArgs& a = P.o;
    a = gemm_base(c, rows_cap, tt);
    a.wmap[0] = Mp.o;
    a.wpk[0] = M.P[l].t[W_O];
    a.x = c->xo; a.x_rows = 2 * c->D.MC;
    a.nseg = 1; a.seg_tile0[0] = 0; a.seg_tile0[1] = d / kTileN; a.seg_rows[0] = d;
    a.w_tiles = d / kTileN;
    a.kc = (qd + kChunkK - 1) / kChunkK;
    a.mode = MODE_RESID;
    a.h = c->h; a.h_ld = d; a.ssq_out = c->ssq;
    a.x_next = c->xd; a.g_next = W.t[W_MLP_NORM];
  }
  // RMSNorm -> gate/up (paired 64-row tiles) -> SiLU(gate) * up
  {
    GemmArgs& a = P.gu;
    a = gemm_base(c, rows_cap, tt_gu);
    a.wmap[0] = Mp.g; a.wmap[1] = Mp.u;
    a.wpk[0] = M.P[l].t[W_G]; a.wpk[1] = M.P[l].t[W_U];
    if (!a.wpk[0] || !a.wpk[1]) a.wpk[0] = a.wpk[1] = nullptr;
    a.x = c->xd; a.x_rows = 2 * c->D.MC;
    a.nseg = 1; a.pair = 1;
    a.w_tiles = (ffn + 63) / 64;
    a.seg_tile0[0] = 0; a.seg_tile0[1] = a.w_tiles; a.seg_rows[0] = ffn;
    a.kc = (d + kChunkK - 1) / kChunkK;
    a.mode = MODE_SWIGLU;
    a.ssq_in = c->ssq; a.ssq_tiles = d / 128; a.inv_d = 1.0f / d; a.eps = cf.rms_eps;
    a.x_next = c->xf;
  }
  // down projection + residual; emits x = h * g_next (next layer's or the final norm)
  {
    GemmArgs& a = P.dn;
    a = gemm_base(c, rows_cap, tt);
    a.wmap[0] = Mp.dn;
    a.wpk[0] = M.P[l].t[W_D];
    a.x = c->xf; a.x_rows = 2 * c->D.MC;
    a.nseg = 1; a.seg_tile0[0] = 0; a.seg_tile0[1] = d / kTileN; a.seg_rows[0] = d;
    a.w_tiles = d / kTileN;
    a.kc = (ffn + kChunkK - 1) / kChunkK;
    a.mode = MODE_RESID;
    a.h = c->h; a.h_ld = d; a.ssq_out = c->ssq;
    a.x_next = c->xd;
    a.g_next = l + 1 < cf.n_layers ? M.L[l + 1].t[W_ATTN_NORM] : M.final_norm;
  }
  return P;
}

// Decoder layers over the current row plan, one launch per phase.
// rows_cap: row capacity of the pass; batch / rows_per_seq: attention work
// decomposition; pt_attn: page table row base the attention kernel indexes
// by its sequence index.
void run_layers(pard_ctx* c, int mi, int rows_cap, int batch, int rows_per_seq, const int* pt_attn,
                cudaStream_t s, int fixed_rows = 0) {
  // Above 64 rows the gate/up projection takes the 128-token tile (one pass
  // over its weights for all rows), the QKV, O and down projections keep
  // 64-token tiles (two passes): they have only 32-48 output tiles, so with
  // 128-token tiles each tile's split-K finish and epilogue (8 chunks) falls
  // on few CTAs and outlasts the bytes saved.
  const int tt_gu = pick_tt(rows_cap);
  const int tt = std::min(tt_gu, 64);
  const AttnGeom geo = attn_geometry(c, mi, rows_per_seq, batch);
  for (int l = 0; l < c->m[mi].cfg.n_layers; ++l) {
    LayerPlan P = layer_plan(c, mi, l, rows_cap, tt, tt_gu, batch, pt_attn, geo, fixed_rows);
    // the pass's row count is written by the embedding kernel, which directly
    // precedes only the first QKV projection
    P.qkv.m_early = l > 0;
    P.o.m_early = P.gu.m_early = P.dn.m_early = 1;
    run_gemm(c, P.qkv, tt, s);
    launch_attention(P.at, geo.groups * geo.n_split, s, true);
    c->launches++;
    run_gemm(c, P.o, tt, s);
    run_gemm(c, P.gu, tt_gu, s);
    run_gemm(c, P.dn, tt, s);
  }
}

// LM head over the packed activation rows x (final-norm scale from ssq_in).
GemmArgs lm_args(pard_ctx* c, int mi, const __nv_bfloat16* x, int x_rows, const float* ssq_in, int rows_cap, int tt,
                 const int* m_dev, float* logits, const int* row_out, const int* row_gi, const int* row_seq,
                 float4* stats, int2* stats_i, int gumbel_stream) {
  Model& M = c->m[mi];
  GemmArgs a = gemm_base(c, rows_cap, tt);
  a.m_dev = m_dev;
  a.wmap[0] = M.lm_map;
  a.wpk[0] = M.lm_pk;
  a.x = x; a.x_rows = x_rows;
  a.nseg = 1;
  a.w_tiles = (M.cfg.vocab + kTileN - 1) / kTileN;
  a.seg_tile0[0] = 0; a.seg_tile0[1] = a.w_tiles; a.seg_rows[0] = M.cfg.vocab;
  a.kc = (M.cfg.d_model + kChunkK - 1) / kChunkK;
  a.mode = MODE_LOGITS;
  a.ssq_in = ssq_in; a.ssq_tiles = M.cfg.d_model / 128; a.inv_d = 1.0f / M.cfg.d_model; a.eps = M.cfg.rms_eps;
  a.logits = logits; a.row_out = row_out; a.row_gi = row_gi; a.row_seq = row_seq;
  a.stats = stats; a.stats_i = stats_i; a.vocab = M.cfg.vocab; a.gumbel_stream = gumbel_stream;
  a.m_early = 1;  // the LM head follows the whole layer stack (or the prefill's gather), far from its row count's writer
  return a;
}

void run_lm_head(pard_ctx* c, int mi, const __nv_bfloat16* x, int x_rows, const float* ssq_in, int rows_cap, int tt,
                 const int* m_dev, float* logits, const int* row_out, const int* row_gi, const int* row_seq,
                 float4* stats, int2* stats_i, int gumbel_stream, cudaStream_t s) {
  GemmArgs a = lm_args(c, mi, x, x_rows, ssq_in, rows_cap, tt, m_dev, logits, row_out, row_gi, row_seq, stats, stats_i,
                       gumbel_stream);
  run_gemm(c, a, tt, s);
}

EmbedArgs embed_base(pard_ctx* c, int mi, int mode) {
  EmbedArgs e;
  std::memset(&e, 0, sizeof(e));
  const Model& M = c->m[mi];
  e.mode = mode;
  e.batch = c->batch; e.K = c->K; e.mask_id = M.cfg.mask_id; e.vocab = M.cfg.vocab; e.d = M.cfg.d_model;
  e.mask_ids = c->n_mask_ids > 0 ? c->mask_ids : nullptr;
  e.embed = M.embed; e.gain0 = M.L[0].t[W_ATTN_NORM];
  e.st = c->st; e.rp = c->rp;
  e.h = c->h; e.x = c->xd; e.ssq = c->ssq; e.m_cap = c->D.MC; e.status = c->status;
  return e;
}

// Move a [N][K] matrix between row-major order and the packed layout, one
// batch of R-row blocks at a time through the workspace scratch.
void pack_matrix(pard_ctx* c, __nv_bfloat16* w, int N, int K, int R, bool unpack, cudaStream_t s) {
  const size_t block = (size_t)R * K;
  const int per_batch = (int)std::max<size_t>(1, kPackTmpBytes / (block * 2));
  __nv_bfloat16* tmp = c->template at<__nv_bfloat16>(c->o.pack_tmp);
  for (int b0 = 0; b0 < N / R; b0 += per_batch) {
    const int nb = std::min(per_batch, N / R - b0);
    CK(cudaMemcpyAsync(tmp, w + (size_t)b0 * block, (size_t)nb * block * 2, cudaMemcpyDeviceToDevice, s));
    launch_pack(tmp, w + (size_t)b0 * block, R, K, nb, unpack, s);
  }
}

template <typename F>
pard_status guarded(F&& f) {
  try {
    return f();
  } catch (const CudaFail& e) {
    return fail(PARD_ERR_CUDA, std::string(e.what) + ": " + cudaGetErrorString(e.e));
  } catch (cudaError_t e) {
    return fail(PARD_ERR_CUDA, std::string("kernel launch: ") + cudaGetErrorString(e));
  } catch (const std::exception& e) {
    return fail(PARD_ERR_CUDA, e.what());
  }
}

}  // namespace

// ============================================================================
// C ABI
// ============================================================================
extern "C" {

const char* pard_last_error(void) { return g_err.c_str(); }

size_t pard_workspace_bytes(const pard_model_cfg* t, const pard_model_cfg* d, const pard_limits* lim) {
  std::string why;
  if (!valid_cfg(t, why) || !valid_cfg(d, why) || !valid_limits(lim, why)) return 0;
  if (t->vocab != d->vocab) return 0;
  // the reduction scratch is sized for the largest GB300 (152 SMs) and below
  Dims D = make_dims(*t, *d, *lim, 160);
  return layout_ws(D, *lim).total;
}

size_t pard_kv_pool_bytes(const pard_model_cfg* t, const pard_model_cfg* d, const pard_limits* lim) {
  std::string why;
  if (!valid_cfg(t, why) || !valid_cfg(d, why) || !valid_limits(lim, why)) return 0;
  return kv_bytes_model(*t, *lim) + kv_bytes_model(*d, *lim);
}

pard_status pard_load_weights(pard_ctx** out, const pard_model_cfg* tcfg, const pard_weights* tw,
                              const pard_model_cfg* dcfg, const pard_weights* dw, const pard_limits* lim,
                              void* kv_pool, size_t kv_pool_bytes, void* workspace, size_t ws_bytes,
                              const int32_t* h_order_t, const int32_t* h_order_d, void* stream) {
  std::string why;
  if (!out) return fail(PARD_ERR_ARG, "null output pointer");
  *out = nullptr;
  if (!valid_cfg(tcfg, why)) return fail(PARD_ERR_SHAPE, "target: " + why);
  if (!valid_cfg(dcfg, why)) return fail(PARD_ERR_SHAPE, "draft: " + why);
  if (!valid_limits(lim, why)) return fail(PARD_ERR_ARG, why);
  if (tcfg->vocab != dcfg->vocab) return fail(PARD_ERR_SHAPE, "target and draft vocabularies differ");
  if (!tw || !dw || !tw->embed || !tw->final_norm || !tw->lm_head || !tw->layers || !dw->embed || !dw->final_norm ||
      !dw->lm_head || !dw->layers)
    return fail(PARD_ERR_ARG, "null weight pointer");
  if (!kv_pool || kv_pool_bytes < pard_kv_pool_bytes(tcfg, dcfg, lim)) return fail(PARD_ERR_ARG, "KV pool too small");
  if (!workspace || ws_bytes < pard_workspace_bytes(tcfg, dcfg, lim)) return fail(PARD_ERR_ARG, "workspace too small");
  if ((reinterpret_cast<uintptr_t>(kv_pool) | reinterpret_cast<uintptr_t>(workspace)) & 255)
    return fail(PARD_ERR_ARG, "KV pool and workspace must be 256-byte aligned");
  for (int mi = 0; mi < 2; ++mi) {
    const int32_t* ord = mi == 0 ? h_order_t : h_order_d;
    if (!ord) continue;
    std::vector<char> seen(lim->n_pages, 0);
    for (int i = 0; i < lim->n_pages; ++i) {
      if (ord[i] < 0 || ord[i] >= lim->n_pages || seen[ord[i]]) return fail(PARD_ERR_ARG, "page order is not a permutation");
      seen[ord[i]] = 1;
    }
  }
  auto check_ptr = [](const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
  const pard_weights* W[2] = {tw, dw};
  const pard_model_cfg* C[2] = {tcfg, dcfg};
  for (int mi = 0; mi < 2; ++mi) {
    if (!check_ptr(W[mi]->embed) || !check_ptr(W[mi]->final_norm) || !check_ptr(W[mi]->lm_head))
      return fail(PARD_ERR_ARG, "weight pointers must be 16-byte aligned");
    for (int i = 0; i < C[mi]->n_layers * 9; ++i)
      if (!check_ptr(W[mi]->layers[i])) return fail(PARD_ERR_ARG, "layer weight pointer null or misaligned");
  }
  pard_ctx* c = new pard_ctx();
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  pard_status st = guarded([&]() -> pard_status {
    int dev = 0;
    CK(cudaGetDevice(&dev));
    CK(cudaDeviceGetAttribute(&c->sm, cudaDevAttrMultiProcessorCount, dev));
    int major = 0, minor = 0;
    CK(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev));
    CK(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev));
    if (major != 10) return fail(PARD_ERR_CUDA, "libpard is compiled for compute capability 10.x (GB300, sm_103a) only");
    c->sm = std::min(c->sm, 160);
    c->lim = *lim;
    c->D = make_dims(*tcfg, *dcfg, *lim, c->sm);
    c->o = layout_ws(c->D, *lim);
    c->ws = reinterpret_cast<uint8_t*>(workspace);
    const WsOffsets& o = c->o;
    c->h = c->at<float>(o.h); c->ssq = c->at<float>(o.ssq); c->ssqg = c->at<float>(o.ssqg); c->q = c->at<float>(o.q);
    c->gpart = c->at<float>(o.gpart);
    c->logits = c->at<float>(o.logits); c->dlogits = c->at<float>(o.dlogits);
    c->xd = c->at<__nv_bfloat16>(o.xd); c->xo = c->at<__nv_bfloat16>(o.xo); c->xf = c->at<__nv_bfloat16>(o.xf);
    c->xg = c->at<__nv_bfloat16>(o.xg);
    c->gcnt = c->at<int>(o.gcnt);
    c->stats_t = c->at<float4>(o.stats_t); c->stats_it = c->at<int2>(o.stats_it);
    c->stats_d = c->at<float4>(o.stats_d); c->stats_id = c->at<int2>(o.stats_id);
    c->rp = RowPlan{c->at<int>(o.row_tok), c->at<int>(o.row_pos), c->at<int>(o.row_seq), c->at<int>(o.row_out),
                    c->at<int>(o.row_gi), c->at<int>(o.seq_row0), c->at<int>(o.m_dev)};
    c->g_row_seq = c->at<int>(o.g_row_seq); c->g_row_gi = c->at<int>(o.g_row_gi); c->g_m = c->at<int>(o.g_m);
    c->st.n = c->at<int>(o.st_n); c->st.pend_cnt = c->at<int>(o.st_pc); c->st.pend = c->at<int>(o.st_pend);
    c->st.gen = c->at<int>(o.st_gen); c->st.max_new = c->at<int>(o.st_max); c->st.done = c->at<int>(o.st_done);
    c->st.d = c->at<int>(o.st_d); c->st.dnorm = c->at<float2>(o.st_dnorm); c->st.samp_a = c->at<int>(o.st_sa);
    c->st.samp_norm = c->at<float4>(o.st_snorm); c->st.samp_part = c->at<float2>(o.st_spart);
    c->st.samp_cnt = c->at<int>(o.st_scnt); c->st.kmax = lim->max_k;
    c->call = c->at<CallArgs>(o.call); c->status = c->at<uint32_t>(o.status);
    c->paths = c->at<uint32_t>(o.paths);

    c->tmp_pos = c->at<int>(o.tmp_pos); c->g_plen = c->at<int>(o.g_plen);
    c->mask_ids = c->at<int>(o.mask_ids);

    // counters start at zero; the reduction kernels leave them at zero
    CK(cudaMemsetAsync(c->gcnt, 0, (size_t)kMaxGemmTiles * 8, s));
    CK(cudaMemsetAsync(c->st.samp_cnt, 0, lim->max_batch * 4, s));
    CK(cudaMemsetAsync(c->status, 0, 4, s));
    CK(cudaMemsetAsync(c->paths, 0, 4, s));
    CK(cudaMemsetAsync(c->xd, 0, (size_t)2 * c->D.MC * c->D.dmax * 2, s));
    CK(cudaMemsetAsync(c->xo, 0, (size_t)2 * c->D.MC * c->D.qdmax * 2, s));
    CK(cudaMemsetAsync(c->xf, 0, (size_t)2 * c->D.MC * c->D.ffn_pad * 2, s));
    CK(cudaMemsetAsync(c->xg, 0, (size_t)2 * c->D.gcap * c->D.dmax * 2, s));

    uint8_t* kvp = reinterpret_cast<uint8_t*>(kv_pool);
    std::vector<int> pt_init((size_t)lim->max_batch * c->D.pt_ld, -1);
    std::set<const void*> packed_set;
    for (int mi = 0; mi < 2; ++mi) {
      Model& M = c->m[mi];
      M.cfg = *C[mi];
      M.embed = reinterpret_cast<const __nv_bfloat16*>(W[mi]->embed);
      M.final_norm = reinterpret_cast<const __nv_bfloat16*>(W[mi]->final_norm);
      M.lm_head = reinterpret_cast<const __nv_bfloat16*>(W[mi]->lm_head);
      M.L.resize(M.cfg.n_layers);
      M.maps.resize(M.cfg.n_layers);
      const int d = M.cfg.d_model, qd = M.qd(), kvd = M.kvd(), ffn = M.cfg.ffn;
      for (int l = 0; l < M.cfg.n_layers; ++l) {
        for (int j = 0; j < 9; ++j) M.L[l].t[j] = reinterpret_cast<const __nv_bfloat16*>(W[mi]->layers[l * 9 + j]);
        LayerMaps& mp = M.maps[l];
        mp.q = make_map(M.L[l].t[W_Q], qd, d, kTileN);
        mp.k = make_map(M.L[l].t[W_K], kvd, d, kTileN);
        mp.v = make_map(M.L[l].t[W_V], kvd, d, kTileN);
        mp.o = make_map(M.L[l].t[W_O], d, qd, kTileN);
        mp.g = make_map(M.L[l].t[W_G], ffn, d, 64);
        mp.u = make_map(M.L[l].t[W_U], ffn, d, 64);
        mp.dn = make_map(M.L[l].t[W_D], d, ffn, kTileN);
      }
      M.lm_map = make_map(M.lm_head, M.cfg.vocab, d, kTileN);
      // pack every matrix whose shape allows it, in place (each matrix once,
      // also when the draft shares the target's tensors)
      M.P.assign(M.cfg.n_layers, LayerW{});
      auto pack = [&](const __nv_bfloat16* w, int N, int K, int R) -> const __nv_bfloat16* {
        if (N % R || K % 64) return nullptr;
        if (!packed_set.count(w)) {
          pack_matrix(c, const_cast<__nv_bfloat16*>(w), N, K, R, false, s);
          packed_set.insert(w);
          c->packed_list.push_back({const_cast<__nv_bfloat16*>(w), R});
          c->packed_shape.push_back({N, K});
        }
        return w;
      };
      for (int l = 0; l < M.cfg.n_layers; ++l) {
        const LayerW& Wl = M.L[l];
        LayerW& Pl = M.P[l];
        for (int j = 0; j < 9; ++j) Pl.t[j] = nullptr;
        Pl.t[W_Q] = pack(Wl.t[W_Q], qd, d, kTileN);
        Pl.t[W_K] = pack(Wl.t[W_K], kvd, d, kTileN);
        Pl.t[W_V] = pack(Wl.t[W_V], kvd, d, kTileN);
        Pl.t[W_O] = pack(Wl.t[W_O], d, qd, kTileN);
        if (ffn % 64 == 0 && d % 64 == 0) {
          Pl.t[W_G] = pack(Wl.t[W_G], ffn, d, 64);
          Pl.t[W_U] = pack(Wl.t[W_U], ffn, d, 64);
        }
        Pl.t[W_D] = pack(Wl.t[W_D], d, ffn, kTileN);
      }
      M.lm_pk = pack(M.lm_head, M.cfg.vocab, d, kTileN);
      CK(cudaStreamSynchronize(s));
      M.kv = reinterpret_cast<__nv_bfloat16*>(kvp);
      M.n_pages_ = lim->n_pages;
      M.page_elems = (size_t)M.cfg.n_kv_heads * lim->page_size * M.cfg.head_dim;
      kvp += kv_bytes_model(M.cfg, *lim);
      M.page_table = c->at<int>(o.pt[mi]);
      CK(cudaMemcpyAsync(M.page_table, pt_init.data(), pt_init.size() * 4, cudaMemcpyHostToDevice, s));
      CK(cudaStreamSynchronize(s));
      // RoPE table: cos / sin of pos * theta^(-2j/hd), computed in double, stored fp32
      const int half = M.cfg.head_dim / 2;
      const int rope_rows = c->D.pt_ld * lim->page_size;  // every position a page can hold
      std::vector<float2> rope((size_t)rope_rows * half);
      for (int p = 0; p < rope_rows; ++p)
        for (int j = 0; j < half; ++j) {
          const double inv = std::pow((double)M.cfg.rope_theta, -2.0 * j / M.cfg.head_dim);
          const double ang = (double)p * inv;
          rope[(size_t)p * half + j] = make_float2((float)std::cos(ang), (float)std::sin(ang));
        }
      M.rope = c->at<float2>(o.rope[mi]);
      CK(cudaMemcpyAsync(M.rope, rope.data(), rope.size() * sizeof(float2), cudaMemcpyHostToDevice, s));
      CK(cudaStreamSynchronize(s));
      c->order[mi].resize(lim->n_pages);
      const int32_t* ord = mi == 0 ? h_order_t : h_order_d;
      for (int i = 0; i < lim->n_pages; ++i) c->order[mi][i] = ord ? ord[i] : i;
    }
    return PARD_OK;
  });
  if (st != PARD_OK) {
    delete c;
    return st;
  }
  *out = c;
  return PARD_OK;
}


pard_status pard_prefill(pard_ctx* c, const int32_t* d_tokens, const int32_t* h_lens, int32_t batch, int32_t n_new,
                         int32_t K, int32_t sample, float temperature, uint64_t seed, int32_t* d_first,
                         void* stream) {
  if (!c || !d_tokens || !h_lens || !d_first) return fail(PARD_ERR_ARG, "null argument");
  if (c->unpacked) return fail(PARD_ERR_STATE, "weights were unpacked; load them again");
  if (batch < 1 || batch > c->lim.max_batch) return fail(PARD_ERR_ARG, "batch outside [1, max_batch]");
  if (K < 0 || K > c->lim.max_k) return fail(PARD_ERR_ARG, "K outside [0, max_k]");
  if (n_new < 1) return fail(PARD_ERR_ARG, "n_new < 1");
  if (sample && !(temperature > 0.f)) return fail(PARD_ERR_ARG, "temperature must be > 0 when sampling");
  const int ps = c->lim.page_size;
  std::vector<int> pages(batch);
  long total_pages = 0;
  for (int b = 0; b < batch; ++b) {
    if (h_lens[b] < 1) return fail(PARD_ERR_ARG, "empty prompt");
    if ((long)h_lens[b] + n_new + 2L * K > c->lim.max_ctx) return fail(PARD_ERR_ARG, "prompt + n_new + 2K exceeds max_ctx");
    pages[b] = (h_lens[b] + n_new + 2 * K + ps - 1) / ps;
    total_pages += pages[b];
  }
  if (total_pages > c->lim.n_pages) return fail(PARD_ERR_NO_PAGES, "KV page pool too small for this batch");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  c->launches = 0;
  return guarded([&]() -> pard_status {
    // page tables: sequences take pages in order from the front of each model's page order
    for (int mi = 0; mi < 2; ++mi) {
      std::vector<int> tbl((size_t)c->lim.max_batch * c->D.pt_ld, -1);
      int at = 0;
      for (int b = 0; b < batch; ++b)
        for (int j = 0; j < pages[b]; ++j) tbl[(size_t)b * c->D.pt_ld + j] = c->order[mi][at++];
      CK(cudaMemcpyAsync(c->m[mi].page_table, tbl.data(), tbl.size() * 4, cudaMemcpyHostToDevice, s));
      CK(cudaStreamSynchronize(s));
    }
    std::vector<int> seqs(c->D.gcap), zeros(c->D.gcap, 0), lens(h_lens, h_lens + batch);
    for (int i = 0; i < c->D.gcap; ++i) seqs[i] = i;
    CK(cudaMemcpyAsync(c->g_row_seq, seqs.data(), seqs.size() * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c->g_row_gi, zeros.data(), zeros.size() * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c->g_m, &batch, 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c->g_plen, lens.data(), lens.size() * 4, cudaMemcpyHostToDevice, s));
    CK(cudaStreamSynchronize(s));
    c->batch = batch;
    c->K = K;
    c->n_new = n_new;
    c->ctx_est.assign(batch, 0);
    for (int b = 0; b < batch; ++b) c->ctx_est[b] = h_lens[b] + n_new;
    c->prefilled = false;
    set_call(c, seed, 0, temperature, sample, s);
    const int chunk = c->lim.prefill_chunk;
    long offset = 0;
    for (int b = 0; b < batch; ++b) {
      const int len = h_lens[b];
      for (int mi = 0; mi < 2; ++mi) {
        Model& M = c->m[mi];
        int last_rows = 0;
        for (int start = 0; start < len; start += chunk) {
          const int rows = std::min(chunk, len - start);
          EmbedArgs e = embed_base(c, mi, EMB_PREFILL);
          e.tokens = d_tokens + offset + start;
          e.pf_seq = b;
          e.pf_pos0 = start;
          e.pf_rows = rows;
          launch_embed(e, rows, s, true);
          c->launches++;
          run_layers(c, mi, rows, 1, rows, M.page_table + (size_t)b * c->D.pt_ld, s);
          last_rows = rows;
        }
        if (mi == 0) {
          launch_gather_rows(c->xd, 2 * c->D.MC, c->ssq, M.cfg.d_model / 128, c->D.MC, last_rows - 1, c->xg,
                             2 * c->D.gcap, c->ssqg, c->D.MC, b, M.cfg.d_model, s, true);
          c->launches++;
        }
      }
      offset += len;
    }
    const int gtt = pick_tt(c->D.gcap);
    run_lm_head(c, 0, c->xg, 2 * c->D.gcap, c->ssqg, batch, gtt, c->g_m, nullptr, nullptr, sample ? c->g_row_gi : nullptr,
                c->g_row_seq, c->stats_t, c->stats_it, STREAM_BONUS, s);
    SelectArgs sa;
    std::memset(&sa, 0, sizeof(sa));
    sa.mode = SEL_FIRST;
    sa.batch = batch; sa.K = K; sa.w_tiles = c->D.w_tiles; sa.m_cap = c->D.MC; sa.vocab = c->D.vocab;
    sa.stats = c->stats_t; sa.stats_i = c->stats_it; sa.call = c->call; sa.st = c->st;
    sa.out = d_first; sa.plen = c->g_plen; sa.n_new = n_new;
    launch_select(sa, s, true);
    c->launches++;
    CK(cudaStreamSynchronize(s));
    CK(cudaGetLastError());
    c->prefilled = true;
    return PARD_OK;
  });
}

pard_status pard_draft(pard_ctx* c, int32_t sample, float temperature, uint64_t seed, uint64_t step, int32_t* d_out,
                       float* d_logits, void* stream) {
  if (!c) return fail(PARD_ERR_ARG, "null context");
  if (!c->prefilled) return fail(PARD_ERR_STATE, "pard_draft before pard_prefill (or after pard_unpack_weights)");
  if (c->K == 0) return fail(PARD_ERR_STATE, "pard_draft with K = 0 (autoregressive decoding has no draft pass)");
  if (c->n_mask_ids > 0 && c->n_mask_ids < c->K - 1)
    return fail(PARD_ERR_STATE, "fewer per-offset mask ids than the K - 1 mask rows of the draft");
  if (sample && !(temperature > 0.f)) return fail(PARD_ERR_ARG, "temperature must be > 0 when sampling");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  c->launches = 0;
  return guarded([&]() -> pard_status {
    set_call(c, seed, step, temperature > 0.f ? temperature : 1.0f, sample, s);
    const int rows_cap = c->batch * 2 * c->K;
    EmbedArgs e = embed_base(c, 1, EMB_DRAFT);
    launch_embed(e, rows_cap, s, true);
    c->launches++;
    Model& M = c->m[1];
    const int keep = (sample || d_logits) ? 1 : 0;
    run_layers(c, 1, rows_cap, c->batch, 2 * c->K, M.page_table, s);
    run_lm_head(c, 1, c->xd, 2 * c->D.MC, c->ssq, rows_cap, pick_tt(rows_cap), c->rp.m_dev,
                keep ? c->dlogits : nullptr, c->rp.row_out, c->rp.row_gi, c->rp.row_seq, c->stats_d, c->stats_id,
                STREAM_DRAFT, s);
    SelectArgs sa;
    std::memset(&sa, 0, sizeof(sa));
    sa.mode = SEL_DRAFT;
    sa.batch = c->batch; sa.K = c->K; sa.w_tiles = c->D.w_tiles; sa.m_cap = c->D.MC; sa.vocab = c->D.vocab;
    sa.stats = c->stats_d; sa.stats_i = c->stats_id; sa.call = c->call; sa.st = c->st;
    sa.seq_row0 = c->rp.seq_row0; sa.out = d_out;
    launch_select(sa, s, true);
    c->launches++;
    if (d_logits)
      CK(cudaMemcpyAsync(d_logits, c->dlogits, (size_t)c->batch * c->K * c->D.vocab * 4, cudaMemcpyDeviceToDevice, s));
    c->last_draft_sampled = sample != 0;
    return PARD_OK;
  });
}

// Vanilla speculative decoding's drafting stage on the same kernels: K
// forward passes of the draft model, pass i picking candidate i (one
// embedding / layers / LM head / select sequence per pass).
pard_status pard_draft_sequential(pard_ctx* c, int32_t sample, float temperature, uint64_t seed, uint64_t step,
                                  int32_t* d_out, float* d_logits, void* stream) {
  if (!c) return fail(PARD_ERR_ARG, "null context");
  if (!c->prefilled) return fail(PARD_ERR_STATE, "pard_draft_sequential before pard_prefill (or after pard_unpack_weights)");
  if (c->K == 0) return fail(PARD_ERR_STATE, "pard_draft_sequential with K = 0 (autoregressive decoding has no draft)");
  if (sample && !(temperature > 0.f)) return fail(PARD_ERR_ARG, "temperature must be > 0 when sampling");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  c->launches = 0;
  return guarded([&]() -> pard_status {
    set_call(c, seed, step, temperature > 0.f ? temperature : 1.0f, sample, s);
    Model& M = c->m[1];
    const int keep = (sample || d_logits) ? 1 : 0;
    for (int i = 0; i < c->K; ++i) {
      // pass 0: the pending real tokens (at most K + 1 per sequence); then one row
      const int per_seq = i == 0 ? c->K + 1 : 1;
      const int rows_cap = c->batch * per_seq;
      EmbedArgs e = embed_base(c, 1, EMB_DRAFT_SEQ);
      e.seq_i = i;
      launch_embed(e, rows_cap, s, true);
      c->launches++;
      run_layers(c, 1, rows_cap, c->batch, per_seq, M.page_table, s);
      run_lm_head(c, 1, c->xd, 2 * c->D.MC, c->ssq, rows_cap, pick_tt(rows_cap), c->rp.m_dev,
                  keep ? c->dlogits : nullptr, c->rp.row_out, c->rp.row_gi, c->rp.row_seq, c->stats_d, c->stats_id,
                  STREAM_DRAFT, s);
      SelectArgs sa;
      std::memset(&sa, 0, sizeof(sa));
      sa.mode = SEL_DRAFT_SEQ;
      sa.seq_i = i;
      sa.batch = c->batch; sa.K = c->K; sa.w_tiles = c->D.w_tiles; sa.m_cap = c->D.MC; sa.vocab = c->D.vocab;
      sa.stats = c->stats_d; sa.stats_i = c->stats_id; sa.call = c->call; sa.st = c->st;
      sa.seq_row0 = c->rp.seq_row0; sa.out = d_out;
      launch_select(sa, s, true);
      c->launches++;
    }
    if (d_logits)
      CK(cudaMemcpyAsync(d_logits, c->dlogits, (size_t)c->batch * c->K * c->D.vocab * 4, cudaMemcpyDeviceToDevice, s));
    c->last_draft_sampled = sample != 0;
    return PARD_OK;
  });
}

pard_status pard_verify(pard_ctx* c, const int32_t* d_draft_in, float temperature, float* d_logits_out,
                        void* stream) {
  if (!c) return fail(PARD_ERR_ARG, "null context");
  if (!c->prefilled) return fail(PARD_ERR_STATE, "pard_verify before pard_prefill");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  c->launches = 0;
  return guarded([&]() -> pard_status {
    set_call(c, 0, 0, temperature > 0.f ? temperature : 1.0f, c->last_draft_sampled ? 1 : 0, s);
    const int rows_cap = c->batch * (c->K + 1);
    EmbedArgs e = embed_base(c, 0, EMB_VERIFY);
    e.d_in = d_draft_in ? d_draft_in : c->st.d;
    if (!d_draft_in && c->st.kmax != c->K) {
      // internal candidates have row pitch kmax; feed them through a packed copy
      for (int b = 0; b < c->batch; ++b)
        CK(cudaMemcpyAsync(c->tmp_pos + b * c->K, c->st.d + b * c->st.kmax, c->K * 4, cudaMemcpyDeviceToDevice, s));
      e.d_in = c->tmp_pos;
    }
    launch_embed(e, rows_cap, s, true);
    c->launches++;
    Model& M = c->m[0];
    // K = 0 (autoregressive) keeps its single row of logits for a sampled accept
    const int keep = (c->last_draft_sampled || d_logits_out || c->K == 0) ? 1 : 0;
    run_layers(c, 0, rows_cap, c->batch, c->K + 1, M.page_table, s, c->K + 1);  // K + 1 rows per sequence
    run_lm_head(c, 0, c->xd, 2 * c->D.MC, c->ssq, rows_cap, pick_tt(rows_cap), c->rp.m_dev,
                keep ? c->logits : nullptr, c->rp.row_out, nullptr, c->rp.row_seq, c->stats_t, c->stats_it,
                STREAM_BONUS, s);
    if (d_logits_out)
      CK(cudaMemcpyAsync(d_logits_out, c->logits, (size_t)c->batch * (c->K + 1) * c->D.vocab * 4,
                         cudaMemcpyDeviceToDevice, s));
    return PARD_OK;
  });
}

pard_status pard_accept_commit(pard_ctx* c, int32_t sample, float temperature, uint64_t seed, uint64_t step,
                               int32_t* d_accept_len, int32_t* d_emitted, int32_t* d_kv_slots, int32_t* d_n_emit,
                               void* stream) {
  if (!c) return fail(PARD_ERR_ARG, "null context");
  if (!c->prefilled) return fail(PARD_ERR_STATE, "pard_accept_commit before pard_prefill");
  if (sample && !(temperature > 0.f)) return fail(PARD_ERR_ARG, "temperature must be > 0 when sampling");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  c->launches = 0;
  return guarded([&]() -> pard_status {
    set_call(c, seed, step, temperature > 0.f ? temperature : 1.0f, sample, s);
    AcceptArgs a;
    std::memset(&a, 0, sizeof(a));
    a.batch = c->batch; a.K = c->K; a.w_tiles = c->D.w_tiles; a.m_cap = c->D.MC; a.vocab = c->D.vocab;
    a.stats = c->stats_t; a.stats_i = c->stats_it; a.logits = c->logits; a.dlogits = c->dlogits;
    a.call = c->call; a.st = c->st;
    a.page_table = c->m[0].page_table; a.pt_ld = c->D.pt_ld; a.page_size = c->lim.page_size;
    a.accept_len = d_accept_len; a.emitted = d_emitted; a.kv_slots = d_kv_slots; a.n_emit = d_n_emit;
    a.status = c->status;
    if (sample) {
      launch_accept_sample(a, s, true);
      c->launches += 2;
    } else {
      launch_accept_greedy(a, s, true);
      c->launches++;
    }
    return PARD_OK;
  });
}

pard_status pard_set_logits(pard_ctx* c, const float* y, const float* z, const int32_t* d, float temperature,
                            void* stream) {
  if (!c || !y || !d) return fail(PARD_ERR_ARG, "null argument");
  if (!c->prefilled) return fail(PARD_ERR_STATE, "pard_set_logits before pard_prefill");
  if (!(temperature > 0.f)) return fail(PARD_ERR_ARG, "temperature must be > 0");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  c->launches = 0;
  return guarded([&]() -> pard_status {
    const int B = c->batch, K = c->K, V = c->D.vocab;
    CK(cudaMemcpyAsync(c->logits, y, (size_t)B * (K + 1) * V * 4, cudaMemcpyDeviceToDevice, s));
    CK(cudaMemcpy2DAsync(c->st.d, c->st.kmax * 4, d, K * 4, K * 4, B, cudaMemcpyDeviceToDevice, s));
    set_call(c, 0, 0, temperature, 1, s);
    launch_row_stats(c->logits, B * (K + 1), V, c->D.w_tiles, c->D.MC, c->call, -1, 1, c->stats_t, c->stats_it, s);
    c->launches++;
    if (z) {
      CK(cudaMemcpyAsync(c->dlogits, z, (size_t)B * K * V * 4, cudaMemcpyDeviceToDevice, s));
      launch_row_stats(c->dlogits, B * K, V, c->D.w_tiles, c->D.MC, c->call, -1, 1, c->stats_d, c->stats_id, s);
      SelectArgs sa;
      std::memset(&sa, 0, sizeof(sa));
      sa.mode = SEL_NORM_ONLY;
      sa.batch = B; sa.K = K; sa.w_tiles = c->D.w_tiles; sa.m_cap = c->D.MC; sa.vocab = V;
      sa.stats = c->stats_d; sa.stats_i = c->stats_id; sa.call = c->call; sa.st = c->st;
      launch_select(sa, s, false);
      c->launches += 2;
    }
    return PARD_OK;
  });
}

pard_status pard_set_draft_logits(pard_ctx* c, const float* z, int32_t sample, float temperature, uint64_t seed,
                                  uint64_t step, int32_t* d_out, void* stream) {
  if (!c || !z || !d_out) return fail(PARD_ERR_ARG, "null argument");
  if (!c->prefilled) return fail(PARD_ERR_STATE, "pard_set_draft_logits before pard_prefill");
  if (c->K == 0) return fail(PARD_ERR_STATE, "pard_set_draft_logits with K = 0 (no draft)");
  if (sample && !(temperature > 0.f)) return fail(PARD_ERR_ARG, "temperature must be > 0 when sampling");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  c->launches = 0;
  return guarded([&]() -> pard_status {
    const int B = c->batch, K = c->K, V = c->D.vocab;
    set_call(c, seed, step, temperature > 0.f ? temperature : 1.0f, sample, s);
    CK(cudaMemcpyAsync(c->dlogits, z, (size_t)B * K * V * 4, cudaMemcpyDeviceToDevice, s));
    launch_row_stats(c->dlogits, B * K, V, c->D.w_tiles, c->D.MC, c->call, STREAM_DRAFT, K, c->stats_d, c->stats_id,
                     s);
    SelectArgs sa;
    std::memset(&sa, 0, sizeof(sa));
    sa.mode = SEL_DRAFT_GIVEN;
    sa.batch = B; sa.K = K; sa.w_tiles = c->D.w_tiles; sa.m_cap = c->D.MC; sa.vocab = V;
    sa.stats = c->stats_d; sa.stats_i = c->stats_id; sa.call = c->call; sa.st = c->st; sa.out = d_out;
    launch_select(sa, s, false);
    c->launches += 2;
    c->last_draft_sampled = sample != 0;
    return PARD_OK;
  });
}

pard_status pard_get_state(pard_ctx* c, int32_t* h_n, int32_t* h_gen, int32_t* h_done, void* stream) {
  if (!c) return fail(PARD_ERR_ARG, "null context");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return guarded([&]() -> pard_status {
    const size_t nb = (size_t)std::max(c->batch, 1) * 4;
    if (h_n) CK(cudaMemcpyAsync(h_n, c->st.n, nb, cudaMemcpyDeviceToHost, s));
    if (h_gen) CK(cudaMemcpyAsync(h_gen, c->st.gen, nb, cudaMemcpyDeviceToHost, s));
    if (h_done) CK(cudaMemcpyAsync(h_done, c->st.done, nb, cudaMemcpyDeviceToHost, s));
    CK(cudaStreamSynchronize(s));
    return PARD_OK;
  });
}

pard_status pard_read_kv(pard_ctx* c, int32_t model, int32_t layer, int32_t b, const int32_t* h_pos, int32_t n,
                         void* d_k, void* d_v, void* stream) {
  if (!c || !h_pos || !d_k || !d_v) return fail(PARD_ERR_ARG, "null argument");
  if (model < 0 || model > 1 || !c->prefilled) return fail(PARD_ERR_ARG, "bad model or no prefill yet");
  const Model& M = c->m[model];
  if (layer < 0 || layer >= M.cfg.n_layers || b < 0 || b >= c->batch || n < 1 || n > 4096)
    return fail(PARD_ERR_ARG, "layer, sequence or count out of range");
  for (int i = 0; i < n; ++i)
    if (h_pos[i] < 0 || h_pos[i] >= c->lim.max_ctx) return fail(PARD_ERR_ARG, "position out of range");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return guarded([&]() -> pard_status {
    std::vector<int> tbl(c->D.pt_ld);
    CK(cudaMemcpyAsync(tbl.data(), M.page_table + (size_t)b * c->D.pt_ld, tbl.size() * 4, cudaMemcpyDeviceToHost, s));
    CK(cudaStreamSynchronize(s));
    for (int i = 0; i < n; ++i)
      if (tbl[h_pos[i] / c->lim.page_size] < 0) return fail(PARD_ERR_ARG, "position has no page");
    CK(cudaMemcpyAsync(c->tmp_pos, h_pos, (size_t)n * 4, cudaMemcpyHostToDevice, s));
    launch_read_kv(M.kcache(layer), M.vcache(layer), M.page_table + (size_t)b * c->D.pt_ld, c->tmp_pos, n,
                   M.cfg.n_kv_heads, M.cfg.head_dim, c->lim.page_size, reinterpret_cast<__nv_bfloat16*>(d_k),
                   reinterpret_cast<__nv_bfloat16*>(d_v), s);
    CK(cudaStreamSynchronize(s));
    return PARD_OK;
  });
}

pard_status pard_last_status(pard_ctx* c, uint32_t* h_flags, void* stream) {
  if (!c || !h_flags) return fail(PARD_ERR_ARG, "null argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return guarded([&]() -> pard_status {
    CK(cudaStreamSynchronize(s));
    CK(cudaMemcpy(h_flags, c->status, 4, cudaMemcpyDeviceToHost));
    CK(cudaMemset(c->status, 0, 4));
    if (*h_flags & (ST_TIMEOUT_TMA | ST_TIMEOUT_MMA | ST_TIMEOUT_EPI))
      return fail(PARD_ERR_TIMEOUT, "a kernel pipeline wait ran out");
    if (*h_flags) return fail(PARD_ERR_DEVICE_CHECK, "a kernel flagged a bad index");
    return PARD_OK;
  });
}

pard_status pard_cod_select(int32_t n, int32_t K, double r, double r_min, uint64_t seed, uint64_t sample_id,
                            int32_t* d_keep, int32_t* d_counts, void* stream) {
  if (n < 1 || n > kCodMaxN) return fail(PARD_ERR_ARG, "COD sample rows outside [1, 4096]");
  if (K < 1 || K > 64) return fail(PARD_ERR_ARG, "COD subtask count outside [1, 64]");
  if (!(r > 0.0 && r <= 1.0) || !(r_min >= 0.0 && r_min <= 1.0))
    return fail(PARD_ERR_ARG, "COD retention r outside (0, 1] or r_min outside [0, 1]");
  if (!d_counts || (K > 1 && !d_keep)) return fail(PARD_ERR_ARG, "null output");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return guarded([&]() -> pard_status {
    launch_cod(n, K, r, r_min, seed, sample_id, d_keep, d_counts, s);
    return PARD_OK;
  });
}

pard_status pard_selftest_stalled_wait(pard_ctx* c, void* stream) {
  if (!c) return fail(PARD_ERR_ARG, "null context");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return guarded([&]() -> pard_status {
    launch_stalled_wait(c->status, s);
    return PARD_OK;
  });
}

pard_status pard_unpack_weights(pard_ctx* c, void* stream) {
  if (!c) return fail(PARD_ERR_ARG, "null context");
  if (c->unpacked) return PARD_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return guarded([&]() -> pard_status {
    for (size_t i = 0; i < c->packed_list.size(); ++i)
      pack_matrix(c, c->packed_list[i].first, c->packed_shape[i].first, c->packed_shape[i].second,
                  c->packed_list[i].second, true, s);
    CK(cudaStreamSynchronize(s));
    c->unpacked = true;
    c->prefilled = false;
    return PARD_OK;
  });
}

int32_t pard_launch_count(pard_ctx* c) { return c ? c->launches : 0; }

pard_status pard_set_mask_ids(pard_ctx* c, const int32_t* h_ids, int32_t n, void* stream) {
  if (!c) return fail(PARD_ERR_ARG, "null context");
  if (!h_ids || n == 0) {
    c->n_mask_ids = 0;
    return PARD_OK;
  }
  if (n < 0 || n > std::max(c->lim.max_k - 1, 0)) return fail(PARD_ERR_ARG, "mask id count outside [0, max_k - 1]");
  for (int i = 0; i < n; ++i)
    if (h_ids[i] < 0 || h_ids[i] >= c->m[1].cfg.vocab) return fail(PARD_ERR_ARG, "mask id outside the draft vocabulary");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return guarded([&]() -> pard_status {
    CK(cudaMemcpyAsync(c->mask_ids, h_ids, (size_t)n * 4, cudaMemcpyHostToDevice, s));
    CK(cudaStreamSynchronize(s));
    c->n_mask_ids = n;
    return PARD_OK;
  });
}

pard_status pard_attention_paths(pard_ctx* c, uint32_t* h_bits, void* stream) {
  if (!c || !h_bits) return fail(PARD_ERR_ARG, "null argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return guarded([&]() -> pard_status {
    CK(cudaStreamSynchronize(s));
    CK(cudaMemcpy(h_bits, c->paths, 4, cudaMemcpyDeviceToHost));
    CK(cudaMemset(c->paths, 0, 4));
    return PARD_OK;
  });
}

pard_status pard_set_attention_split_cap(pard_ctx* c, int32_t cap) {
  if (!c) return fail(PARD_ERR_ARG, "null context");
  if (cap < 0 || cap > kMaxAttnSplit) return fail(PARD_ERR_ARG, "attention split cap outside [0, 16]");
  c->attn_split_cap = cap == 0 ? kMaxAttnSplit : cap;
  return PARD_OK;
}

void pard_destroy(pard_ctx* c) { delete c; }

}  // extern "C"
