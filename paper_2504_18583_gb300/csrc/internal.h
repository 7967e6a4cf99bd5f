// Host-side structures shared by the translation units of libpard.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/pard.h"

namespace pard {

constexpr int kTileN = 128;     // weight rows per UMMA tile (MMA M)
constexpr int kChunkK = 64;     // K elements per pipeline stage (one 128-byte swizzle row)
constexpr int kEpiTok = 16;     // tokens per epilogue pass (32 TMEM columns: hi/lo pairs)
constexpr int kMaxSeg = 3;

enum GemmMode : int { MODE_QKV = 0, MODE_RESID = 1, MODE_SWIGLU = 2, MODE_LOGITS = 3 };

// Per-call scalars kept in device memory, so that captured launches read the
// current call's values.
struct CallArgs {
  uint64_t seed;
  uint64_t step;
  float temp;
  int32_t sample;
  int32_t K;
  int32_t pad;
};

struct GemmArgs {
  CUtensorMap wmap[kMaxSeg];  // row-major weights (A operand) for shapes that are not packed;
                              // pair mode: [0] gate, [1] up, 64-row boxes
  const __nv_bfloat16* wpk[kMaxSeg];  // packed weights (null: use wmap)
  const __nv_bfloat16* x;     // packed activations (B operand): row 2m = hi(m), 2m+1 = lo(m)
  int x_rows;                 // rows of the activation buffer (2 x row capacity)
  int nseg;
  int seg_tile0[kMaxSeg + 1]; // prefix sums of tiles per segment
  int seg_rows[kMaxSeg];      // rows of each segment
  int pair;
  int w_tiles, tok_tiles, kc;
  int n_tok;                  // token rows a tile's MMA covers (multiple of 8, <= the tile; 0: the whole tile):
                              // a single-tile pass of fewer rows loads and multiplies only those
  int m_early;                // m_dev was written two or more launches back: read it before the PDL wait and
                              // skip the token tiles past it (0: process every tile)
  int mode;
  int m_cap;                  // row capacity of the activation/output buffers
  const int* m_dev;           // runtime row count
  float* partials;
  int* counters;              // split-K arrival masks: 64-bit word per output tile, zero between launches
  uint32_t* status;
  int stages;                 // ring slots used (0: all the kernel has)
  int pre_stages;             // slots filled before waiting on the previous kernel (0: stages)
  // RMS row scale applied after the reduction (null: none)
  const float* ssq_in;
  int ssq_tiles;
  float inv_d, eps;
  // MODE_RESID
  float* h;
  int h_ld;
  float* ssq_out;
  __nv_bfloat16* x_next;      // packed, x_rows rows
  const __nv_bfloat16* g_next;
  // MODE_QKV
  float* q_out;
  int q_ld;
  __nv_bfloat16* kcache;
  __nv_bfloat16* vcache;
  const int* page_table;
  int pt_ld;
  const int* row_pos;
  const int* row_seq;
  const float2* rope;
  int hd, hkv, page_size, n_pages;
  // MODE_LOGITS
  float* logits;              // [rows_out][vocab] or null
  const int* row_out;         // row -> output row, -1: none (null: identity)
  const int* row_gi;          // row -> Philox row index for Gumbel draws, -1: none
  float4* stats;              // [w_tiles][m_cap] {max, sumexp(T), gumbel best, 0}
  int2* stats_i;              // [w_tiles][m_cap] {argmax, gumbel argmax}
  int vocab;
  int gumbel_stream;
  const CallArgs* call;
};

struct AttnArgs {
  const float* q;             // [rows][hq*hd] fp32, post-RoPE
  int q_ld;
  const __nv_bfloat16* kcache;
  const __nv_bfloat16* vcache;
  const int* page_table;
  int pt_ld;
  const int* row_pos;
  const int* seq_row0;        // [B+1] first row of each sequence in this pass
  int rows_per_seq;           // > 0: every sequence has this many rows (row0 = b x it), seq_row0 unread
  const int* m_dev;
  int batch;
  int hq, hkv, hd, page_size, n_pages;
  int row_blocks;             // row blocks per sequence (grid.y / ...)
  int n_split;                // key splits
  int nbuf;                   // K/V chunk buffers a CTA keeps (4, or 2 for ragged or crowded passes)
  float scale;
  __nv_bfloat16* x_out;       // packed [2*rows][hq*hd] hi/lo
  int x_rows;
  uint32_t* status;
  uint32_t* paths;            // combine paths taken (kAttnPath* bits, OR-ed; null: not recorded)
};

// Attention combine paths recorded in AttnArgs::paths: push or pull combine
// of the key splits, and bit kAttnPathSplit0 + n for clusters of n CTAs.
constexpr uint32_t kAttnPathPush = 1u << 0;
constexpr uint32_t kAttnPathPull = 1u << 1;
constexpr uint32_t kAttnPathRing2 = 1u << 2;  // the two-buffer K/V ring variant ran
constexpr int kAttnPathSplit0 = 3;


// Per-sequence decode state, in the workspace.
struct DevState {
  int* n;          // [B] tokens so far, the pending one included (target cache holds n-1)
  int* pend_cnt;   // [B] draft tokens waiting to be fed (a+1 after a commit)
  int* pend;       // [B][kmax+1]
  int* gen;        // [B] tokens generated (counted toward max_new)
  int* max_new;    // [B]
  int* done;       // [B]
  int* d;          // [B][kmax] current candidates
  float2* dnorm;   // [B][kmax] draft row (max logit, sum exp) at the draft temperature
  int* samp_a;     // [B] sampling: first rejected index (K: all accepted)
  float4* samp_norm;  // [B] (max_y, S_y, max_z, S_z) of the rejected row
  float2* samp_part;  // [B][kResampleSplit] (score, index) partial draws
  int* samp_cnt;      // [B]
  int kmax;        // row pitch of pend (kmax+1) and d (kmax)
};

constexpr int kResampleSplit = 32;

struct RowPlan {     // row layout of one forward pass
  int* row_tok;
  int* row_pos;
  int* row_seq;
  int* row_out;      // logits output row or -1
  int* row_gi;       // Philox row index for Gumbel draws or -1
  int* seq_row0;     // [B+1]
  int* m_dev;
};

struct EmbedArgs {
  int mode;          // EMB_PREFILL, EMB_DRAFT, EMB_VERIFY, EMB_DRAFT_SEQ
  int batch, K, mask_id, vocab, d;
  int seq_i;         // EMB_DRAFT_SEQ: pass index i (0: the pending tokens; i > 0: candidate i-1)
  const int* mask_ids;  // EMB_DRAFT: id of mask m_k per offset k (null: mask_id for all)
  const __nv_bfloat16* embed;
  const __nv_bfloat16* gain0;  // first layer's attention-norm gain
  const int* tokens;           // prefill: this chunk's tokens
  int pf_seq, pf_pos0, pf_rows;
  const int* d_in;             // verify: candidates to feed ([B][K])
  DevState st;
  RowPlan rp;
  float* h;
  __nv_bfloat16* x;            // packed, 2 * m_cap rows
  float* ssq;
  int m_cap;
  uint32_t* status;
};
enum { EMB_PREFILL = 0, EMB_DRAFT = 1, EMB_VERIFY = 2, EMB_DRAFT_SEQ = 3 };

struct SelectArgs {
  int mode;          // SEL_DRAFT, SEL_FIRST, SEL_NORM_ONLY, SEL_DRAFT_SEQ, SEL_DRAFT_GIVEN
  int batch, K, w_tiles, m_cap, vocab;
  int seq_i;         // SEL_DRAFT_SEQ: the candidate this pass picks
  const float4* stats;
  const int2* stats_i;
  const CallArgs* call;
  DevState st;
  const int* seq_row0;
  int* out;          // draft: [B][K]; first token: [B]
  const int* plen;   // first token: prompt lengths
  int n_new;
};
// SEL_DRAFT_GIVEN: candidates from given draft logits rows b * K + i
enum { SEL_DRAFT = 0, SEL_FIRST = 1, SEL_NORM_ONLY = 2, SEL_DRAFT_SEQ = 3, SEL_DRAFT_GIVEN = 4 };

struct AcceptArgs {
  int batch, K, w_tiles, m_cap, vocab;
  const float4* stats;
  const int2* stats_i;
  const float* logits;     // [B][K+1][V] (sampling)
  const float* dlogits;    // [B][K][V] (sampling)
  const CallArgs* call;
  DevState st;
  const int* page_table;
  int pt_ld, page_size;
  int* accept_len;
  int* emitted;
  int* kv_slots;
  int* n_emit;
  uint32_t* status;        // sticky device status word (null: none)
};

constexpr int kMaxGemmTiles = 32768;  // output tiles (weight tile x token tile) of one GEMM launch
constexpr int kMaxQVRows = 64;          // query vectors of one attention work unit
constexpr int kMaxAttnSplit = 16;       // key splits (CTAs of one cluster) of one attention work unit

// launchers (gemm.cu, attention.cu, misc.cu)
void launch_embed(const EmbedArgs& a, int grid, cudaStream_t s, bool pdl);
void launch_gather_rows(const __nv_bfloat16* x, int x_rows, const float* ssq, int ssq_tiles, int m_cap_src, int src_row,
                        __nv_bfloat16* xg, int xg_rows, float* ssqg, int m_cap_dst, int dst_row, int d, cudaStream_t s,
                        bool pdl);
void launch_pack(const __nv_bfloat16* tmp, __nv_bfloat16* w, int R, int K, int nblocks, bool unpack, cudaStream_t s);
void launch_select(const SelectArgs& a, cudaStream_t s, bool pdl);
void launch_accept_greedy(const AcceptArgs& a, cudaStream_t s, bool pdl);
void launch_accept_sample(const AcceptArgs& a, cudaStream_t s, bool pdl);
void launch_row_stats(const float* logits, int rows, int vocab, int w_tiles, int m_cap, const CallArgs* call,
                      int gumbel_stream, int rows_per_seq, float4* stats, int2* stats_i, cudaStream_t s);
void launch_set_call(CallArgs* dst, CallArgs v, cudaStream_t s, bool pdl);
void launch_copy_i32(const int* src, int* dst, int n, cudaStream_t s, bool pdl);
void launch_copy_f32(const float* src, float* dst, size_t n, cudaStream_t s, bool pdl);
void launch_read_kv(const __nv_bfloat16* kc, const __nv_bfloat16* vc, const int* page_table_row, const int* pos, int n,
                    int hkv, int hd, int page_size, __nv_bfloat16* ok, __nv_bfloat16* ov, cudaStream_t s);

void launch_stalled_wait(uint32_t* status, cudaStream_t s);
constexpr int kCodMaxN = 4096;  // rows per subtask of one COD sample
void launch_cod(int N, int K, double r, double r_min, uint64_t seed, uint64_t sample_id, int32_t* keep,
                int32_t* counts, cudaStream_t s);
void launch_gemm(const GemmArgs& a, int tt, int grid, cudaStream_t s, bool pdl);
int gemm_smem_bytes(int tt);
void launch_attention(const AttnArgs& a, int grid_x, cudaStream_t s, bool pdl);
int attention_rows_per_block(int group);

}  // namespace pard
