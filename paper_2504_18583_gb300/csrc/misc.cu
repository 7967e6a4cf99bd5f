// Small kernels of the decode step: row planning + embedding gather, the
// draft's token selection from LM-head statistics, acceptance with KV
// commit / rollback, and helpers for tests.
#include <algorithm>
#include <climits>

#include "common.cuh"
#include "internal.h"

namespace pard {

#define PARD_LAUNCH(kernel, grid, block, smem, strm, pdl, ...)                       \
  do {                                                                                 \
    cudaLaunchConfig_t cfg_ = {};                                                      \
    cfg_.gridDim = dim3(grid);                                                         \
    cfg_.blockDim = dim3(block);                                                       \
    cfg_.dynamicSmemBytes = (smem);                                                    \
    cfg_.stream = (strm);                                                              \
    cudaLaunchAttribute at_[1];                                                        \
    at_[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;                    \
    at_[0].val.programmaticStreamSerializationAllowed = 1;                             \
    cfg_.attrs = at_;                                                                  \
    cfg_.numAttrs = (pdl) ? 1 : 0;                                                     \
    cudaError_t e_ = cudaLaunchKernelEx(&cfg_, kernel, __VA_ARGS__);                   \
    if (e_ != cudaSuccess) throw e_;                                                   \
  } while (0)

// ---------------------------------------------------------------------------
// Row plan + embedding.  One block per row of the pass (grid = row capacity).
//   draft  (Eq. 6): sequence b feeds its pend_cnt pending real tokens, then
//                   K-1 mask tokens (one shared id, or one id per offset),
//                   at positions n-p .. n+K-2; logits rows are the last real
//                   row and every mask row;
//   verify:         [last token, d_0..d_{K-1}] at positions n-1 .. n+K-1;
//   sequential draft (vanilla speculative decoding), pass i: i = 0 feeds
//                   the pending real tokens (logits row: the last), i > 0
//                   feeds candidate d_{i-1} at position n-1+i;
//   prefill:        a chunk of one sequence's prompt.
// h = E[token]; x = h * g (hi/lo bf16 pairs); ssq[t][m] = sum of h^2 over
// the 128 columns of tile t.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(128) embed_kernel(const __grid_constant__ EmbedArgs a) {
  pdl_wait();
  pdl_trigger();
  __shared__ int s_row0[65];
  __shared__ int s_tok;
  const int m = blockIdx.x;
  if (threadIdx.x == 0) {
    int total = 0;
    if (a.mode == EMB_PREFILL) {
      s_row0[0] = 0;
      total = a.pf_rows;
    } else {
      for (int b = 0; b < a.batch; ++b) {
        s_row0[b] = total;
        total += a.mode == EMB_DRAFT       ? a.st.pend_cnt[b] + a.K - 1
                 : a.mode == EMB_DRAFT_SEQ ? (a.seq_i == 0 ? a.st.pend_cnt[b] : 1)
                                           : a.K + 1;
      }
      s_row0[a.batch] = total;
    }
    if (m == 0) {
      *a.rp.m_dev = total;
      if (a.mode == EMB_PREFILL) { a.rp.seq_row0[0] = 0; a.rp.seq_row0[1] = total; }
      else for (int b = 0; b <= a.batch; ++b) a.rp.seq_row0[b] = s_row0[b];
      if (total > a.m_cap) set_status(a.status, ST_BAD_ROWS);
    }
    s_tok = -1;
    if (m < total && m < a.m_cap) {
      int b = 0, j = m, tok = 0, pos = 0, out = -1, gi = -1;
      if (a.mode == EMB_PREFILL) {
        b = a.pf_seq;
        tok = a.tokens[m];
        pos = a.pf_pos0 + m;
      } else {
        while (b + 1 < a.batch && m >= s_row0[b + 1]) ++b;
        j = m - s_row0[b];
        const int n = a.st.n[b];
        if (a.mode == EMB_DRAFT) {
          const int p = a.st.pend_cnt[b];
          tok = j < p ? a.st.pend[b * (a.st.kmax + 1) + j] : (a.mask_ids ? a.mask_ids[j - p] : a.mask_id);
          pos = n - p + j;
          if (j >= p - 1) { gi = j - (p - 1); out = b * a.K + gi; }
        } else if (a.mode == EMB_DRAFT_SEQ) {
          const int p = a.st.pend_cnt[b];
          if (a.seq_i == 0) {
            tok = a.st.pend[b * (a.st.kmax + 1) + j];
            pos = n - p + j;
            if (j == p - 1) { gi = 0; out = b * a.K; }
          } else {
            tok = a.st.d[b * a.st.kmax + a.seq_i - 1];
            pos = n - 1 + a.seq_i;
            gi = a.seq_i;
            out = b * a.K + a.seq_i;
          }
        } else {
          tok = j == 0 ? a.st.pend[b * (a.st.kmax + 1) + a.st.pend_cnt[b] - 1] : a.d_in[b * a.K + j - 1];
          if (j > 0) a.st.d[b * a.st.kmax + j - 1] = tok;
          pos = n - 1 + j;
          out = b * (a.K + 1) + j;
        }
      }
      if (tok < 0 || tok >= a.vocab) { set_status(a.status, ST_BAD_TOKEN); tok = 0; }
      a.rp.row_tok[m] = tok;
      a.rp.row_pos[m] = pos;
      a.rp.row_seq[m] = b;
      a.rp.row_out[m] = out;
      a.rp.row_gi[m] = gi;
      s_tok = tok;
    }
  }
  __syncthreads();
  const int tok = s_tok;
  if (tok < 0) return;
  const __nv_bfloat16* e = a.embed + (size_t)tok * a.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int t = warp; t < a.d / 128; t += 4) {
    float ss = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int c = t * 128 + lane * 4 + k;
      const float h = __bfloat162float(e[c]);
      a.h[(size_t)m * a.d + c] = h;
      __nv_bfloat16 hi, lo;
      split_bf16(h * __bfloat162float(a.gain0[c]), hi, lo);
      a.x[xpk(2 * m, c, 2 * a.m_cap)] = hi;
      a.x[xpk(2 * m + 1, c, 2 * a.m_cap)] = lo;
      ss += h * h;
    }
    ss = warp_sum(ss);
    if (lane == 0) a.ssq[(size_t)t * a.m_cap + m] = ss;
  }
}

// Failure-path self test: one thread waits, through the pipelines' bounded
// wait, on an mbarrier that nothing arrives on; the wait gives up after its
// limit (kWaitLimitNs) and flags ST_TIMEOUT_TMA, as a stalled pipeline would,
// and the kernel returns normally.
__global__ void stalled_wait_kernel(uint32_t* status) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int never_raised;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  never_raised = 0;
  fence_barrier_init();
  if (!mbar_wait(&bar, 0, &never_raised)) set_status(status, ST_TIMEOUT_TMA);
}

void launch_stalled_wait(uint32_t* status, cudaStream_t s) {
  PARD_LAUNCH(stalled_wait_kernel, 1, 32, 0, s, false, status);
}

void launch_embed(const EmbedArgs& a, int grid, cudaStream_t s, bool pdl) {
  PARD_LAUNCH(embed_kernel, grid, 128, 0, s, pdl, a);
}

// Copy one activation row (hi/lo pair, packed layout) and its sum-of-squares partials.
__global__ void gather_rows_kernel(const __nv_bfloat16* x, int x_rows, const float* ssq, int ssq_tiles, int m_cap_src,
                                   int src_row, __nv_bfloat16* xg, int xg_rows, float* ssqg, int m_cap_dst, int dst_row,
                                   int d) {
  pdl_wait();
  pdl_trigger();
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    xg[xpk(2 * dst_row, c, xg_rows)] = x[xpk(2 * src_row, c, x_rows)];
    xg[xpk(2 * dst_row + 1, c, xg_rows)] = x[xpk(2 * src_row + 1, c, x_rows)];
  }
  for (int t = threadIdx.x; t < ssq_tiles; t += blockDim.x)
    ssqg[(size_t)t * m_cap_dst + dst_row] = ssq[(size_t)t * m_cap_src + src_row];
}

void launch_gather_rows(const __nv_bfloat16* x, int x_rows, const float* ssq, int ssq_tiles, int m_cap_src, int src_row,
                        __nv_bfloat16* xg, int xg_rows, float* ssqg, int m_cap_dst, int dst_row, int d, cudaStream_t s,
                        bool pdl) {
  PARD_LAUNCH(gather_rows_kernel, 1, 256, 0, s, pdl, x, x_rows, ssq, ssq_tiles, m_cap_src, src_row, xg, xg_rows, ssqg,
              m_cap_dst, dst_row, d);
}

// Weight packing: nblocks consecutive R-row blocks of a [N][K] matrix move
// between row-major order and the packed layout ([K/64][R][64] per block,
// 16-byte chunks of row r rotated by r mod 8).  tmp holds a copy of the
// blocks in the source order; w is overwritten in the destination order.
__global__ void pack_kernel(const __nv_bfloat16* tmp, __nv_bfloat16* w, int R, int K, int nblocks, int unpack) {
  const int kc = K / 64;
  const size_t chunks = (size_t)nblocks * R * kc * 8;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < chunks; i += (size_t)gridDim.x * blockDim.x) {
    const int j = (int)(i % 8);
    size_t t = i / 8;
    const int kk = (int)(t % kc);
    t /= kc;
    const int r = (int)(t % R);
    const size_t b = t / R;
    const size_t rm = (b * R + r) * (size_t)K + (size_t)kk * 64 + (size_t)j * 8;
    const size_t pk = ((b * kc + kk) * R + r) * 64 + (size_t)((j ^ (r & 7)) << 3);
    if (!unpack)
      *reinterpret_cast<uint4*>(w + pk) = *reinterpret_cast<const uint4*>(tmp + rm);
    else
      *reinterpret_cast<uint4*>(w + rm) = *reinterpret_cast<const uint4*>(tmp + pk);
  }
}

void launch_pack(const __nv_bfloat16* tmp, __nv_bfloat16* w, int R, int K, int nblocks, bool unpack, cudaStream_t s) {
  const size_t chunks = (size_t)nblocks * R * (K / 64) * 8;
  const int grid = (int)std::min<size_t>((chunks + 255) / 256, 4096);
  PARD_LAUNCH(pack_kernel, grid, 256, 0, s, false, tmp, w, R, K, nblocks, unpack ? 1 : 0);
}

// ---------------------------------------------------------------------------
// Reductions of the LM-head tile statistics.
// (max, sum exp((x - max)/T)) pairs merge by rescaling to the larger max.
// ---------------------------------------------------------------------------
struct RowRed {
  float mx; int arg; float se; float gv; int gi;
};

__device__ __forceinline__ void merge_lse(float& m1, float& s1, float m2, float s2, float T) {
  if (m2 == -INFINITY) return;
  if (m1 == -INFINITY) { m1 = m2; s1 = s2; return; }
  const float M = fmaxf(m1, m2);
  s1 = s1 * expf(m1 / T - M / T) + s2 * expf(m2 / T - M / T);
  m1 = M;
}

__device__ __forceinline__ void merge_red(RowRed& r, const RowRed& o, float T) {
  float m1 = r.mx, s1 = r.se;
  merge_lse(m1, s1, o.mx, o.se, T);
  float v = r.mx;
  int i = r.arg;
  argmax_merge(v, i, o.mx, o.arg);
  r.arg = i;
  r.mx = m1;
  r.se = s1;
  argmax_merge(r.gv, r.gi, o.gv, o.gi);
}

// Block-wide reduction over the w_tiles tile statistics of one row; every
// thread returns the result.  Fixed order: strided per thread, then a tree.
__device__ RowRed reduce_row(const float4* stats, const int2* stats_i, int w_tiles, int m_cap, int m, float T,
                             RowRed* sred) {
  RowRed r{-INFINITY, INT_MAX, 0.f, -INFINITY, INT_MAX};
  for (int t = threadIdx.x; t < w_tiles; t += blockDim.x) {
    const float4 s = stats[(size_t)t * m_cap + m];
    const int2 si = stats_i[(size_t)t * m_cap + m];
    RowRed o{s.x, si.x, s.y, s.z, si.y < 0 ? INT_MAX : si.y};
    merge_red(r, o, T);
  }
  sred[threadIdx.x] = r;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) merge_red(sred[threadIdx.x], sred[threadIdx.x + w], T);
    __syncthreads();
  }
  RowRed out = sred[0];
  __syncthreads();
  return out;
}

// Draft tokens (argmax or Gumbel-max winner) and draft-row normalisers;
// or the prefill's first token and state initialisation.
__global__ void __launch_bounds__(256) select_kernel(const __grid_constant__ SelectArgs a) {
  pdl_wait();
  pdl_trigger();
  __shared__ RowRed sred[256];
  const float T = a.call->temp;
  const bool sample = a.call->sample != 0;
  int b, i = 0, m;
  if (a.mode == SEL_FIRST) {
    b = blockIdx.x;
    m = b;
  } else if (a.mode == SEL_DRAFT_SEQ) {
    b = blockIdx.x;
    i = a.seq_i;
    m = i == 0 ? a.seq_row0[b] + a.st.pend_cnt[b] - 1 : b;
  } else {
    b = blockIdx.x / a.K;
    i = blockIdx.x % a.K;
    m = a.mode == SEL_DRAFT ? a.seq_row0[b] + a.st.pend_cnt[b] - 1 + i : b * a.K + i;
  }
  const RowRed r = reduce_row(a.stats, a.stats_i, a.w_tiles, a.m_cap, m, T, sred);
  if (threadIdx.x != 0) return;
  const int tok = sample ? r.gi : r.arg;
  if (a.mode == SEL_FIRST) {
    a.out[b] = tok;
    const int kp = a.st.kmax + 1;
    a.st.n[b] = a.plen[b] + 1;
    a.st.pend_cnt[b] = 1;
    a.st.pend[b * kp] = tok;
    a.st.gen[b] = 1;
    a.st.max_new[b] = a.n_new;
    a.st.done[b] = a.n_new <= 1 ? 1 : 0;
    return;
  }
  a.st.dnorm[b * a.st.kmax + i] = make_float2(r.mx, r.se);
  if (a.mode == SEL_DRAFT || a.mode == SEL_DRAFT_SEQ || a.mode == SEL_DRAFT_GIVEN) {
    a.st.d[b * a.st.kmax + i] = tok;
    if (a.out) a.out[b * a.K + i] = tok;
  }
}

void launch_select(const SelectArgs& a, cudaStream_t s, bool pdl) {
  const int grid = (a.mode == SEL_FIRST || a.mode == SEL_DRAFT_SEQ) ? a.batch : a.batch * a.K;
  PARD_LAUNCH(select_kernel, grid, 256, 0, s, pdl, a);
}

// ---------------------------------------------------------------------------
// Commit / rollback of one sequence (a accepted candidates + one bonus).
// ---------------------------------------------------------------------------
__device__ void commit_seq(const AcceptArgs& a, int b, int acc, const int* emitted_tok) {
  const int K = a.K, kp = a.st.kmax + 1;
  if (a.st.done[b]) {
    if (a.accept_len) a.accept_len[b] = 0;
    if (a.n_emit) a.n_emit[b] = 0;
    for (int j = 0; j <= K; ++j) {
      if (a.emitted) a.emitted[b * (K + 1) + j] = -1;
      if (a.kv_slots) a.kv_slots[b * (K + 1) + j] = -1;
    }
    return;
  }
  const int n = a.st.n[b];
  const int room = a.st.max_new[b] - a.st.gen[b];
  const int take = acc + 1 < room ? acc + 1 : room;
  for (int j = 0; j <= K; ++j) {
    if (a.emitted) a.emitted[b * (K + 1) + j] = j < take ? emitted_tok[j] : -1;
    if (a.kv_slots) {
      int slot = -1;
      if (j <= acc) {
        const int pos = n - 1 + j;
        slot = a.page_table[(size_t)b * a.pt_ld + pos / a.page_size] * a.page_size + pos % a.page_size;
      }
      a.kv_slots[b * (K + 1) + j] = slot;
    }
  }
  for (int j = 0; j <= acc; ++j) a.st.pend[b * kp + j] = emitted_tok[j];
  a.st.pend_cnt[b] = acc + 1;
  a.st.n[b] = n + acc + 1;
  a.st.gen[b] += take;
  if (a.st.gen[b] >= a.st.max_new[b]) a.st.done[b] = 1;
  if (a.accept_len) a.accept_len[b] = acc;
  if (a.n_emit) a.n_emit[b] = take;
}

// Greedy: a = longest prefix with d_i == argmax y_i, bonus = argmax y_a.
__global__ void __launch_bounds__(256) accept_greedy_kernel(const __grid_constant__ AcceptArgs a) {
  pdl_wait();
  pdl_trigger();
  __shared__ RowRed sred[256];
  __shared__ int s_arg[17];
  const int b = blockIdx.x;
  for (int i = 0; i <= a.K; ++i) {
    const RowRed r = reduce_row(a.stats, a.stats_i, a.w_tiles, a.m_cap, b * (a.K + 1) + i, 1.0f, sred);
    if (threadIdx.x == 0) s_arg[i] = r.arg;
  }
  if (threadIdx.x != 0) return;
  int acc = 0;
  while (acc < a.K && a.st.d[b * a.st.kmax + acc] == s_arg[acc]) ++acc;
  // a candidate outside the vocabulary never equals an argmax (rejected); flag it
  for (int i = 0; i < a.K && a.status; ++i) {
    const int di = a.st.d[b * a.st.kmax + i];
    if (di < 0 || di >= a.vocab) set_status(a.status, ST_BAD_TOKEN);
  }
  int em[17];
  for (int j = 0; j < acc; ++j) em[j] = a.st.d[b * a.st.kmax + j];
  em[acc] = s_arg[acc];
  commit_seq(a, b, acc, em);
}

void launch_accept_greedy(const AcceptArgs& a, cudaStream_t s, bool pdl) {
  PARD_LAUNCH(accept_greedy_kernel, a.batch, 256, 0, s, pdl, a);
}

// Sampling, phase 1: row normalisers and the accept tests
// u_i * q_i(d_i) < p_i(d_i), p = softmax(y/T), q = softmax(z/T).
__global__ void __launch_bounds__(256) accept_test_kernel(const __grid_constant__ AcceptArgs a) {
  pdl_wait();
  pdl_trigger();
  __shared__ RowRed sred[256];
  __shared__ float2 s_norm[17];
  const int b = blockIdx.x;
  const float T = a.call->temp;
  for (int i = 0; i <= a.K; ++i) {
    const RowRed r = reduce_row(a.stats, a.stats_i, a.w_tiles, a.m_cap, b * (a.K + 1) + i, T, sred);
    if (threadIdx.x == 0) s_norm[i] = make_float2(r.mx, r.se);
  }
  if (threadIdx.x != 0) return;
  int j = a.K;
  for (int i = 0; i < a.K; ++i) {
    const int di = a.st.d[b * a.st.kmax + i];
    if (di < 0 || di >= a.vocab) {
      // a candidate outside the vocabulary has no probability: rejected
      if (a.status) set_status(a.status, ST_BAD_TOKEN);
      j = i;
      break;
    }
    const float yv = a.logits[((size_t)b * (a.K + 1) + i) * a.vocab + di];
    const float p = expf(yv / T - s_norm[i].x / T) / s_norm[i].y;
    const float2 zn = a.st.dnorm[b * a.st.kmax + i];
    const float zv = a.dlogits[((size_t)b * a.K + i) * a.vocab + di];
    const float q = expf(zv / T - zn.x / T) / zn.y;
    const float u = uniform01(philox_word(a.call->seed, STREAM_ACCEPT, a.call->step, (uint32_t)b, (uint32_t)i, 0u));
    if (!(u * q < p)) { j = i; break; }
  }
  a.st.samp_a[b] = j;
  const float2 zn = j < a.K ? a.st.dnorm[b * a.st.kmax + j] : make_float2(0.f, 1.f);
  a.st.samp_norm[b] = make_float4(s_norm[j].x, s_norm[j].y, zn.x, zn.y);
}

// Sampling, phase 2: the bonus token by Gumbel-max over the vocabulary,
// from max(0, p_j - q_j) at the first rejection j, or from p_K; split over
// kResampleSplit blocks per sequence, the last one merges in block order
// and commits.
__global__ void __launch_bounds__(256) resample_kernel(const __grid_constant__ AcceptArgs a) {
  pdl_wait();
  pdl_trigger();
  __shared__ float s_v[256];
  __shared__ int s_i[256];
  __shared__ int s_last;
  const int b = blockIdx.x / kResampleSplit, part = blockIdx.x % kResampleSplit;
  const float T = a.call->temp;
  const int j = a.st.samp_a[b];
  const float4 nm = a.st.samp_norm[b];
  const float* y = a.logits + ((size_t)b * (a.K + 1) + j) * a.vocab;
  const float* z = j < a.K ? a.dlogits + ((size_t)b * a.K + j) * a.vocab : nullptr;
  const int v0 = (int)((long)part * a.vocab / kResampleSplit), v1 = (int)((long)(part + 1) * a.vocab / kResampleSplit);
  float best = -INFINITY;
  int bi = INT_MAX;
  for (int v = v0 + threadIdx.x; v < v1; v += blockDim.x) {
    const float g = gumbel(philox_word(a.call->seed, STREAM_BONUS, a.call->step, (uint32_t)b, 0u, (uint32_t)v));
    float sc;
    if (z) {
      const float p = expf(y[v] / T - nm.x / T) / nm.y;
      const float q = expf(z[v] / T - nm.z / T) / nm.w;
      const float w = fmaxf(p - q, 0.f);
      sc = w > 0.f ? logf(w) + g : -INFINITY;
    } else {
      sc = y[v] / T + g;
    }
    argmax_merge(best, bi, sc, v);
  }
  s_v[threadIdx.x] = best;
  s_i[threadIdx.x] = bi;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) {
      float v = s_v[threadIdx.x];
      int i = s_i[threadIdx.x];
      argmax_merge(v, i, s_v[threadIdx.x + w], s_i[threadIdx.x + w]);
      s_v[threadIdx.x] = v;
      s_i[threadIdx.x] = i;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    a.st.samp_part[b * kResampleSplit + part] = make_float2(s_v[0], __int_as_float(s_i[0]));
    __threadfence();
    const int old = atomicAdd(&a.st.samp_cnt[b], 1);
    s_last = old == kResampleSplit - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  float gbest = -INFINITY;
  int gi = INT_MAX;
  if (threadIdx.x == 0) {
    for (int p = 0; p < kResampleSplit; ++p) {
      const float2 pv = __ldcg(&a.st.samp_part[b * kResampleSplit + p]);
      argmax_merge(gbest, gi, pv.x, __float_as_int(pv.y));
    }
    a.st.samp_cnt[b] = 0;
    s_i[0] = gi;
    s_v[0] = gbest;
  }
  __syncthreads();
  if (s_v[0] == -INFINITY) {
    // max(0, p - q) vanished everywhere (p == q up to rounding): draw from p_j
    float bb = -INFINITY;
    int bj = INT_MAX;
    for (int v = threadIdx.x; v < a.vocab; v += blockDim.x) {
      const float g = gumbel(philox_word(a.call->seed, STREAM_BONUS, a.call->step, (uint32_t)b, 0u, (uint32_t)v));
      const float p = expf(y[v] / T - nm.x / T) / nm.y;
      argmax_merge(bb, bj, logf(p) + g, v);
    }
    __syncthreads();
    s_v[threadIdx.x] = bb;
    s_i[threadIdx.x] = bj;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
      if ((int)threadIdx.x < w) {
        float v = s_v[threadIdx.x];
        int i = s_i[threadIdx.x];
        argmax_merge(v, i, s_v[threadIdx.x + w], s_i[threadIdx.x + w]);
        s_v[threadIdx.x] = v;
        s_i[threadIdx.x] = i;
      }
      __syncthreads();
    }
  }
  if (threadIdx.x != 0) return;
  int em[17];
  for (int k = 0; k < j; ++k) em[k] = a.st.d[b * a.st.kmax + k];
  em[j] = s_i[0];
  commit_seq(a, b, j, em);
}

void launch_accept_sample(const AcceptArgs& a, cudaStream_t s, bool pdl) {
  PARD_LAUNCH(accept_test_kernel, a.batch, 256, 0, s, pdl, a);
  PARD_LAUNCH(resample_kernel, a.batch * kResampleSplit, 256, 0, s, true, a);
}

// Tile statistics of given logits rows (same layout as the LM-head
// epilogue): per 128-entry tile the max and argmax, the sum of exp((x - max)/T)
// and, when gumbel_stream >= 0 and the call samples, the Gumbel-max winner of
// the tile for row m = b * rows_per_seq + i (Philox row i of sequence b), the
// draw the LM-head epilogue makes for a draft row.
__global__ void __launch_bounds__(128) row_stats_kernel(const float* logits, int vocab, int m_cap, const CallArgs* call,
                                                        int gumbel_stream, int rows_per_seq, float4* stats,
                                                        int2* stats_i) {
  pdl_wait();
  const int t = blockIdx.x, m = blockIdx.y;
  const int v = t * 128 + threadIdx.x;
  const float T = call->temp;
  const bool valid = v < vocab;
  const bool gumb = gumbel_stream >= 0 && call->sample != 0;
  const float x = valid ? logits[(size_t)m * vocab + v] : -INFINITY;
  __shared__ float s_v[4], s_g[4];
  __shared__ int s_i[4], s_gi[4];
  __shared__ float s_m;
  float mv = x;
  int mi = valid ? v : INT_MAX;
  warp_argmax(mv, mi);
  float gv = -INFINITY;
  int gi = INT_MAX;
  if (gumb && valid) {
    gv = gumbel_score(x, T, call->seed, (uint32_t)gumbel_stream, call->step, (uint32_t)(m / rows_per_seq),
                      (uint32_t)(m % rows_per_seq), (uint32_t)v);
    gi = v;
  }
  if (gumb) warp_argmax(gv, gi);
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) { s_v[w] = mv; s_i[w] = mi; s_g[w] = gv; s_gi[w] = gi; }
  __syncthreads();
  if (threadIdx.x == 0) {
    float bv = s_v[0];
    int bi = s_i[0];
    for (int k = 1; k < 4; ++k) argmax_merge(bv, bi, s_v[k], s_i[k]);
    float bg = s_g[0];
    int bgi = s_gi[0];
    for (int k = 1; k < 4; ++k) argmax_merge(bg, bgi, s_g[k], s_gi[k]);
    s_m = bv;
    s_i[0] = bi;
    s_g[0] = bg;
    s_gi[0] = bgi;
  }
  __syncthreads();
  const float mxv = s_m;
  const int arg = s_i[0];
  float e = valid ? expf(x / T - mxv / T) : 0.f;
  e = warp_sum(e);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) s_v[w] = e;
  __syncthreads();
  if (threadIdx.x == 0) {
    stats[(size_t)t * m_cap + m] =
        make_float4(mxv, ((s_v[0] + s_v[1]) + s_v[2]) + s_v[3], gumb ? s_g[0] : -INFINITY, 0.f);
    stats_i[(size_t)t * m_cap + m] = make_int2(arg, gumb ? s_gi[0] : -1);
  }
}

void launch_row_stats(const float* logits, int rows, int vocab, int w_tiles, int m_cap, const CallArgs* call,
                      int gumbel_stream, int rows_per_seq, float4* stats, int2* stats_i, cudaStream_t s) {
  PARD_LAUNCH(row_stats_kernel, dim3(w_tiles, rows), 128, 0, s, false, logits, vocab, m_cap, call, gumbel_stream,
              rows_per_seq > 0 ? rows_per_seq : 1, stats, stats_i);
}

__global__ void set_call_kernel(CallArgs* dst, CallArgs v) {
  pdl_wait();
  pdl_trigger();
  *dst = v;
}
void launch_set_call(CallArgs* dst, CallArgs v, cudaStream_t s, bool pdl) {
  PARD_LAUNCH(set_call_kernel, 1, 1, 0, s, pdl, dst, v);
}

__global__ void copy_i32_kernel(const int* src, int* dst, int n) {
  pdl_wait();
  pdl_trigger();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) dst[i] = src[i];
}
void launch_copy_i32(const int* src, int* dst, int n, cudaStream_t s, bool pdl) {
  PARD_LAUNCH(copy_i32_kernel, 1, 256, 0, s, pdl, src, dst, n);
}

__global__ void copy_f32_kernel(const float4* src, float4* dst, size_t n4) {
  pdl_wait();
  pdl_trigger();
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4; i += (size_t)gridDim.x * blockDim.x)
    dst[i] = src[i];
}
void launch_copy_f32(const float* src, float* dst, size_t n, cudaStream_t s, bool pdl) {
  // n is a multiple of 4 and both pointers are 16-byte aligned (checked by the caller)
  const size_t n4 = n / 4;
  int grid = (int)((n4 + 255) / 256);
  if (grid > 1216) grid = 1216;
  if (grid < 1) grid = 1;
  PARD_LAUNCH(copy_f32_kernel, grid, 256, 0, s, pdl, reinterpret_cast<const float4*>(src),
              reinterpret_cast<float4*>(dst), n4);
}

__global__ void read_kv_kernel(const __nv_bfloat16* kc, const __nv_bfloat16* vc, const int* pt, const int* pos, int n,
                               int hkv, int hd, int ps, __nv_bfloat16* ok, __nv_bfloat16* ov) {
  const int i = blockIdx.x;
  if (i >= n) return;
  const int p = pos[i];
  const int page = pt[p / ps];
  for (int e = threadIdx.x; e < hkv * hd; e += blockDim.x) {
    const int h = e / hd, c = e % hd;
    const size_t off = (((size_t)page * hkv + h) * ps + p % ps) * hd + c;
    ok[(size_t)i * hkv * hd + e] = kc[off];
    ov[(size_t)i * hkv * hd + e] = vc[off];
  }
}
void launch_read_kv(const __nv_bfloat16* kc, const __nv_bfloat16* vc, const int* page_table_row, const int* pos, int n,
                    int hkv, int hd, int page_size, __nv_bfloat16* ok, __nv_bfloat16* ov, cudaStream_t s) {
  PARD_LAUNCH(read_kv_kernel, n, 128, 0, s, false, kc, vc, page_table_row, pos, n, hkv, hd, page_size, ok, ov);
}

}  // namespace pard
