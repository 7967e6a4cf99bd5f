/*
 * libpard -- PARD speculative decode step on one GB300 (sm_103a).
 *
 * C ABI: plain pointers and sizes only.  Pointers named d_* are device
 * pointers, h_* are host pointers.  `stream` is a cudaStream_t passed as
 * void*; every call that takes one only enqueues work on it (no host
 * synchronisation) unless stated otherwise.  No call allocates device memory:
 * the caller owns the weights, the KV page pool and the workspace, sized by
 * pard_kv_pool_bytes / pard_workspace_bytes; the library only borrows them.
 * Errors are returned as pard_status codes, with a message available from
 * pard_last_error(); kernels that detect a bad index or a stalled pipeline
 * set a sticky device status word read by pard_last_status().
 *
 * The decode step (paper: PARD, arXiv 2504.18583):
 *   pard_draft          one draft forward over the accepted prefix plus
 *                       mask tokens predicts K tokens at once (Section 3.1,
 *                       Eq. 6; shared mask id, Section 4.3)
 *   pard_verify         one target forward over the last token and the K
 *                       candidates (Section 2.2, verification stage)
 *   pard_accept_commit  greedy prefix match or speculative-sampling
 *                       rejection with residual resampling (the rule of the
 *                       speculative decoding papers the paper builds on,
 *                       Section 2.2), then KV commit / rollback by length
 * pard_prefill fills both caches from the prompts and emits the first token.
 */
#ifndef PARD_H
#define PARD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  PARD_OK = 0,
  PARD_ERR_ARG = -1,          /* null pointer, bad size or bad value */
  PARD_ERR_SHAPE = -2,        /* model shape the kernels do not support */
  PARD_ERR_NO_PAGES = -3,     /* KV page pool too small for the request */
  PARD_ERR_CUDA = -4,         /* a CUDA runtime/driver call failed */
  PARD_ERR_DEVICE_CHECK = -5, /* a kernel flagged a bad index (see pard_last_status) */
  PARD_ERR_TIMEOUT = -6,      /* a kernel pipeline wait ran out (see pard_last_status) */
  PARD_ERR_STATE = -7         /* call out of order (e.g. draft before prefill) */
} pard_status;

/* Llama-style decoder shape (the LLaMA3 family of Section 4.1).
 * Supported: head_dim 64 or 128, n_q_heads a multiple of n_kv_heads,
 * d_model, n_q_heads*head_dim and n_kv_heads*head_dim multiples of 128,
 * ffn a multiple of 8, vocab a multiple of 8, mask_id in [0, vocab). */
typedef struct {
  int32_t n_layers, d_model, n_q_heads, n_kv_heads, head_dim, ffn, vocab;
  float rope_theta, rms_eps;
  int32_t mask_id;
} pard_model_cfg;

/* Device pointers to bf16 weights, all row-major [out][in]:
 *   embed [vocab][d], final_norm [d], lm_head [vocab][d],
 *   layers: host array of n_layers*9 device pointers, per layer in the order
 *   attn_norm [d], wq [hq*hd][d], wk [hkv*hd][d], wv [hkv*hd][d],
 *   wo [d][hq*hd], mlp_norm [d], wg [ffn][d], wu [ffn][d], wd [d][ffn].
 * Every pointer must be 16-byte aligned.  Borrowed until pard_destroy. */
typedef struct {
  const void* embed;
  const void* final_norm;
  const void* lm_head;
  const void* const* layers;
} pard_weights;

/* Sizes the workspace and page pool are built for. */
typedef struct {
  int32_t max_batch;      /* sequences decoded together (<= 64) */
  int32_t max_k;          /* draft length K (1..16) */
  int32_t max_ctx;        /* positions one sequence may reach (prompt + new + 2K) */
  int32_t page_size;      /* KV page size in tokens (16) */
  int32_t prefill_chunk;  /* rows per prefill forward (multiple of 64, <= 1024) */
  int32_t n_pages;        /* pages in each model's pool */
} pard_limits;

typedef struct pard_ctx pard_ctx;

/* Bytes of device workspace needed for these models and limits (host only,
 * no CUDA call).  Returns 0 if the arguments are invalid. */
size_t pard_workspace_bytes(const pard_model_cfg* target, const pard_model_cfg* draft, const pard_limits* lim);

/* Bytes of the KV page pool: lim->n_pages pages for each model, each page
 * holding K and V of page_size tokens for every layer, bf16, laid out
 * [layer][K|V][page][kv_head][token][head_dim].  Host only. */
size_t pard_kv_pool_bytes(const pard_model_cfg* target, const pard_model_cfg* draft, const pard_limits* lim);

/* Loads the two models of the method: the target model that verifies and the
 * PARD draft model that proposes K tokens per forward pass (Section 3.1).
 * Section 4.1 trains the smallest variant of a model series as the draft of
 * that series' targets (e.g. the LLaMA3.1-8B and LLaMA3.3-70B rows of
 * Table 1); both are Llama-style decoders with bf16 weights.  The caller owns
 * the weights, the KV page pool and the workspace; the library borrows them
 * until pard_destroy.
 * Validate shapes, record the borrowed pointers, carve the workspace and
 * build TMA descriptors and RoPE tables.
 * IN-PLACE PACKING: every projection and LM-head matrix whose row count is a
 * multiple of 128 (64 for wg/wu) and whose column count is a multiple of 64
 * is rearranged in place into 128-row x 64-column blocks (64-row for wg/wu),
 * each stored contiguously with its 16-byte chunks rotated by (row mod 8), so
 * that one weight tile is one contiguous 16 KB copy.  The bytes stay inside
 * each matrix's own allocation; a matrix shared by both models is packed
 * once.  pard_unpack_weights restores row-major order.  The embedding and
 * the norm gains are never moved.  h_page_order_{target,draft}
 * (host, n_pages entries each, a permutation of 0..n_pages-1, or NULL for
 * the identity) give the order in which pages are handed to sequences.
 * Synchronises `stream` once (uploads tables).  On success *out owns host
 * state only; device memory stays the caller's. */
pard_status pard_load_weights(pard_ctx** out, const pard_model_cfg* target, const pard_weights* target_w,
                              const pard_model_cfg* draft, const pard_weights* draft_w, const pard_limits* lim,
                              void* d_kv_pool, size_t kv_pool_bytes, void* d_workspace, size_t workspace_bytes,
                              const int32_t* h_page_order_target, const int32_t* h_page_order_draft, void* stream);

/* Prefill both models on `batch` prompts (d_tokens: the prompts
 * concatenated, h_lens[b] tokens each) and emit each sequence's first new
 * token into d_first_token[b].  This is the prompt pass that precedes the
 * decode iterations of Section 2.2: it fills the target's and the draft's KV
 * caches with the prompt (the prefix key-value states the draft and verify
 * passes attend to) and the target's last-row logits give x_n, the first
 * token that the first draft pass extends (argmax, or a Gumbel-max draw at
 * `temperature` with Philox stream 2, step 0 when sample != 0).
 * Reserves ceil((len + n_new + 2K) / page_size) pages per sequence and
 * model, in sequence order, from the front of the page order.
 * n_new: tokens to generate per sequence, the first one included; K: the
 * draft length every later pard_draft uses.  K = 0 selects autoregressive
 * decoding with the target alone (Eq. 2): each pard_verify runs one row per
 * sequence and pard_accept_commit emits its argmax (or a draw from it), and
 * pard_draft returns PARD_ERR_STATE; it is the baseline the paper's speedups
 * are measured against.  Synchronises `stream`. */
pard_status pard_prefill(pard_ctx* ctx, const int32_t* d_tokens, const int32_t* h_lens, int32_t batch,
                         int32_t n_new, int32_t K, int32_t sample, float temperature, uint64_t seed,
                         int32_t* d_first_token, void* stream);

/* One draft forward (Eq. 6): the pending real tokens of each sequence, then
 * K-1 mask tokens, at consecutive positions; the K predictions are read at
 * the last real row and at every mask row.  Greedy: argmax; sample != 0:
 * Gumbel-max draw from softmax(z / temperature) with Philox stream 0.
 * Writes d_draft_out [B][K] and, if non-NULL, the draft logits
 * d_draft_logits [B][K][vocab] (fp32).  Mask rows leave the draft cache by
 * length only. */
pard_status pard_draft(pard_ctx* ctx, int32_t sample, float temperature, uint64_t seed, uint64_t step,
                       int32_t* d_draft_out, float* d_draft_logits, void* stream);

/* Vanilla speculative decoding's drafting stage (Section 2.2: the draft
 * model produces the K candidates autoregressively; Section 3.1's
 * autoregressive factorization), on the same kernels: K draft forwards,
 * pass 0 over the pending real tokens (candidate 0 read at the last row),
 * pass i >= 1 over candidate i-1 alone at position n-1+i.  Same arguments,
 * outputs, sampling streams (Philox stream 0, row i for candidate i) and
 * errors as pard_draft, and the same commit afterwards (the pending tokens
 * are fed again next step), so pard_verify / pard_accept_commit follow it
 * unchanged.  Per iteration it costs K draft forwards against PARD's one:
 * the comparison of the paper's two iteration times, K*T_D + T_T and
 * T_D + T_T. */
pard_status pard_draft_sequential(pard_ctx* ctx, int32_t sample, float temperature, uint64_t seed, uint64_t step,
                                  int32_t* d_draft_out, float* d_draft_logits, void* stream);

/* Per-offset mask ids for the parallel draft (Section 4.3 compares one
 * shared mask id with distinct ones): mask m_k (k = 0 .. K-2) takes
 * h_ids[k]; h_ids = NULL or n = 0 restores the draft config's shared
 * mask_id.  n <= max_k - 1, ids in [0, draft vocab); a later pard_draft
 * with K - 1 > n returns PARD_ERR_STATE.  Synchronises `stream`. */
pard_status pard_set_mask_ids(pard_ctx* ctx, const int32_t* h_ids, int32_t n, void* stream);

/* One target forward over [last token, d_0..d_{K-1}] at positions
 * n-1..n+K-1 of each sequence.  d_draft_in [B][K]: candidates to verify, or
 * NULL for the ones the last pard_draft produced.  Writes per-row logit
 * statistics for pard_accept_commit and, if non-NULL, the logits
 * d_logits_out [B][K+1][vocab] (fp32). */
pard_status pard_verify(pard_ctx* ctx, const int32_t* d_draft_in, float temperature, float* d_logits_out,
                        void* stream);

/* Accept and commit.  Greedy: a = longest prefix with d_i == argmax y_i,
 * bonus = argmax y_a.  sample != 0: accept d_i while u_i * q_i(d_i) <
 * p_i(d_i) (u_i: Philox stream 1), at the first rejection j draw the bonus
 * from max(0, p_j - q_j) renormalised, after K acceptances draw it from p_K
 * (Gumbel-max, stream 2).  Then target length += a + 1 (rejected slots are
 * dropped by length), draft pending tokens = d_0..d_{a-1}, bonus.
 * Outputs (device, may be NULL): d_accept_len [B] = a; d_emitted [B][K+1]
 * = emitted tokens that count toward n_new, -1 after them; d_kv_slots
 * [B][K+1] = cache slots page*page_size + pos%page_size of the committed
 * target positions n-1..n-1+a, -1 after them; d_n_emit [B] = tokens counted.
 * Finished sequences keep their state and report a = 0, no tokens. */
pard_status pard_accept_commit(pard_ctx* ctx, int32_t sample, float temperature, uint64_t seed, uint64_t step,
                               int32_t* d_accept_len, int32_t* d_emitted, int32_t* d_kv_slots, int32_t* d_n_emit,
                               void* stream);

/* Replace the logits the next pard_accept_commit reads (testing the
 * acceptance rule on given inputs): d_target_logits [B][K+1][vocab],
 * d_draft_logits [B][K][vocab] (may be NULL when greedy), d_draft [B][K].
 * A candidate outside [0, vocab) is rejected at its offset and flags
 * ST_BAD_TOKEN in the device status word. */
pard_status pard_set_logits(pard_ctx* ctx, const float* d_target_logits, const float* d_draft_logits,
                            const int32_t* d_draft, float temperature, void* stream);

/* Candidates from given draft logits (testing the draft pass's token
 * selection, Eq. 6, on identical inputs): d_draft_logits [B][K][vocab] take
 * the place of the logits pard_draft reads at its K prediction rows;
 * candidate d_i = argmax z_i, or (sample != 0) the Gumbel-max draw from
 * softmax(z_i / temperature) with Philox stream 0, row i -- the selection
 * pard_draft makes from its LM head's tile statistics.  The candidates, the
 * logits and their row normalisers become the ones the next pard_verify /
 * pard_accept_commit use.  Writes d_draft_out [B][K]. */
pard_status pard_set_draft_logits(pard_ctx* ctx, const float* d_draft_logits, int32_t sample, float temperature,
                                  uint64_t seed, uint64_t step, int32_t* d_draft_out, void* stream);

/* Host copy of per-sequence state: h_n [B] (tokens so far, incl. pending),
 * h_generated [B], h_done [B].  Synchronises `stream`.  Any may be NULL. */
pard_status pard_get_state(pard_ctx* ctx, int32_t* h_n, int32_t* h_generated, int32_t* h_done, void* stream);

/* Copy one layer's KV entries at the given positions of sequence b into
 * host-visible device buffers d_k, d_v [n][n_kv_heads][head_dim] (bf16),
 * reading through the page table (for checking the cache layout).
 * model: 0 target, 1 draft. */
pard_status pard_read_kv(pard_ctx* ctx, int32_t model, int32_t layer, int32_t b, const int32_t* h_pos, int32_t n,
                         void* d_k, void* d_v, void* stream);

/* Synchronise `stream` and return the sticky device status word in
 * *h_flags (0 = clean); the word is cleared.  Returns PARD_ERR_TIMEOUT or
 * PARD_ERR_DEVICE_CHECK when bits are set. */
pard_status pard_last_status(pard_ctx* ctx, uint32_t* h_flags, void* stream);

/* COD data construction (Section 3.2, appendix algorithm) for one training
 * sample of n+1 tokens and K subtasks: d_keep[(k-2)*n + j] = 1 when row j of
 * mask subtask k (k = 2..K; position j, fed mask m_{k-2}, labelled x_{j+1})
 * is kept, and d_counts[k-1] = rows kept by subtask k (d_counts[0] = n:
 * subtask 1, ordinary next-token training, keeps every row).  Subtask k keeps
 * round(n * max(r^(k-1), r_min)) rows (r^(k-1) by repeated multiplication in
 * double, half up), chosen among the rows whose predecessor (row j-1 of
 * subtask k-1) is kept -- the integrity of prefix key-value states; every
 * subtask-2 row qualifies, rows j < k-2 never do.  The choice keeps the
 * candidates with the smallest Philox words (stream 3, step = sample_id,
 * row k, v = j; ties to the lower j), so it is reproducible.  Bounds:
 * 1 <= n <= 4096, 1 <= K <= 64, 0 < r <= 1, 0 <= r_min <= 1; d_keep holds
 * (K-1)*n int32 (may be NULL when K = 1), d_counts K int32, both device
 * memory.  Needs no context; enqueues one kernel on `stream`. */
pard_status pard_cod_select(int32_t n, int32_t K, double r, double r_min, uint64_t seed, uint64_t sample_id,
                            int32_t* d_keep, int32_t* d_counts, void* stream);

/* Failure-path self test: enqueue one kernel whose bounded pipeline wait
 * (the one every GEMM stage uses) waits on a barrier nothing completes; after
 * the wait limit (2 s) it sets the timeout bit of the device status word
 * (bit 0) and returns, leaving the context usable.  A following
 * pard_last_status returns PARD_ERR_TIMEOUT with that bit. */
pard_status pard_selftest_stalled_wait(pard_ctx* ctx, void* stream);

/* Restore every matrix pard_load_weights packed to row-major order
 * (synchronises `stream`).  The context accepts no further decode calls. */
pard_status pard_unpack_weights(pard_ctx* ctx, void* stream);

/* Acceptance from given logits, allocating nothing.  The paper has no
 * counterpart: this is an interface for callers that cannot provide device
 * memory of their own -- runtimes without a device allocator, or engines that
 * plan all device memory ahead and forbid allocation on their serving path.
 * Inputs and outputs are as for pard_set_logits + pard_accept_commit (the
 * same kernels, same results): d_target_logits [batch][K+1][vocab],
 * d_draft_logits [batch][K][vocab] (needed only when sample != 0), d_draft
 * [batch][K]; outputs d_accept_len [batch] and d_emitted [batch][K+1] (-1
 * after the emitted tokens).  A candidate outside [0, vocab) is never read
 * from the logits: it counts as a rejection at its offset.  Nothing is
 * committed anywhere: no context is involved.
 * Scratch: one fixed file-scope device array of about 6.3 MiB, sized for
 * batch <= 16, 1 <= K <= 8, vocab <= 128256 (vocab a multiple of 8); larger
 * sizes return PARD_ERR_ARG with a message.  Every GPU that loads the
 * library keeps that array until the process exits.  The first call on a
 * device looks up the array's device address (cudaGetSymbolAddress, with that
 * device current) and caches it; make that first call before any stream
 * capture.  All calls share the array and each call re-initialises the state
 * it needs (including the counters that must start at zero), so calls whose
 * work overlaps on the GPU race: issue them on one stream. */
pard_status pard_accept_noalloc(const float* d_target_logits, const float* d_draft_logits, const int32_t* d_draft,
                                int32_t batch, int32_t K, int32_t vocab, int32_t sample, float temperature,
                                uint64_t seed, uint64_t step, int32_t* d_accept_len, int32_t* d_emitted,
                                void* stream);

/* Kernel launches the last call enqueued (for launch accounting). */
int32_t pard_launch_count(pard_ctx* ctx);

/* Diagnostics of the attention kernel (Section 2.2: the verify pass attends
 * over the full prefix; Eq. 6: so does the draft pass).  The key range of
 * one (sequence, kv head, row block) unit is split over the CTAs of one
 * thread-block cluster, whose partial results are combined either by a push
 * into each finishing CTA's shared memory (when the receive area fits beside
 * the CTAs' key/value buffers: short contexts) or by a pull over distributed
 * shared memory (long contexts).  pard_attention_paths synchronises `stream`
 * and returns in *h_bits which forms ran since the last read (bit 0: push,
 * bit 1: pull, bit 2: the two-buffer K/V ring that passes with ragged
 * contexts or with more multi-chunk units than two per SM take, bit 3 + n: a
 * cluster of n CTAs), then clears the record.
 * pard_set_attention_split_cap limits the key splits of one unit to cap
 * CTAs (1..16; 0 restores the default 16) from the next pass on: the
 * launcher falls back to 8-CTA clusters on a GPU that cannot place 16, and a
 * cap gives that form on any GPU.  Both return PARD_ERR_ARG for a null
 * context or a cap outside [0, 16]. */
pard_status pard_attention_paths(pard_ctx* ctx, uint32_t* h_bits, void* stream);
pard_status pard_set_attention_split_cap(pard_ctx* ctx, int32_t cap);

/* Thread-local message for the last failing call ("" if none). */
const char* pard_last_error(void);

/* Release host state.  Does not free caller-owned device memory. */
void pard_destroy(pard_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* PARD_H */
