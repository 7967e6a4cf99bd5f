// Weight-streaming GEMM for the decode step: Y[m][n] = sum_k X[m][k] W[n][k]
// with W bf16 [N][K] streamed from HBM exactly once per launch and X a few
// activation rows (M = K+1 verify rows, up to 2K draft rows per sequence).
//
// GB300 design (one CTA per SM, persistent, stream-K):
//  * operand swap: the weight tile is the UMMA A operand (M = 128 weight
//    rows), the activations the B operand (N = 2 x token tile), so a skinny
//    M=9 product still issues full 128-row tensor-core tiles;
//  * activations are carried as bf16 hi/lo pairs (x = hi + lo, rows 2m and
//    2m+1 of the B operand), which keeps fp32-level accuracy of the products
//    with bf16 tensor-core inputs; hi and lo columns are summed in the
//    epilogue;
//  * warp 0 streams 128x64 weight tiles and the matching activation tile
//    with TMA (128-byte swizzle) through a multi-stage mbarrier ring, warp 1
//    issues tcgen05.mma into a TMEM accumulator, warps 2-5 drain TMEM;
//  * the flattened (tile, K-chunk) index space is split evenly over the
//    CTAs; a tile shared by several CTAs is finished by the last one to
//    arrive, which sums the partials in CTA order (deterministic);
//  * epilogues are fused: RMS row scaling, RoPE + paged KV write (QKV),
//    residual add + next norm's gain and sum of squares (O / down),
//    SiLU(gate) * up (gate/up pairs), logits + per-tile max / argmax /
//    sum-exp / Gumbel-max statistics (LM head);
//  * programmatic dependent launch: the weight tiles of the first stages
//    are requested before waiting on the previous kernel, since weights do
//    not depend on it.
#include <climits>

#include "common.cuh"
#include "internal.h"

namespace pard {

template <int TT>
struct GemmCfg {
  static constexpr int kABytes = kTileN * 128;       // 128 rows x 64 bf16
  static constexpr int kBBytes = 2 * TT * 128;       // 2*TT rows x 64 bf16
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStages = TT <= 16 ? 5 : (TT <= 32 ? 4 : 3);
  static constexpr int kAccCols = 2 * TT;
  static constexpr int kNumAcc = (2 * kAccCols <= 256) ? 2 : 1;
  static constexpr int kTmemCols = kNumAcc * kAccCols <= 32 ? 32 : kNumAcc * kAccCols <= 64 ? 64
                                   : kNumAcc * kAccCols <= 128 ? 128 : 256;
  static constexpr int kChunks = TT / kEpiTok;
  // scratch after the stage ring
  static constexpr int kBarBytes = 8 * (2 * kStages + 4);
  static constexpr int kMiscBytes = 64;
  static constexpr int kScratchFloats = TT + 4 * 64 + 16 + kEpiTok * kTileN;
  static constexpr int kSmem = 1024 + kStages * kStageBytes + kBarBytes + kMiscBytes + 4 * kScratchFloats;
};

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

__device__ __forceinline__ long owner_of(long u, long U, long G) { return ((u + 1) * G + U - 1) / U - 1; }
__device__ __forceinline__ long range_start(long c, long U, long G) { return c * U / G; }

__device__ __forceinline__ int seg_of(const GemmArgs& a, int w_tile) {
  int s = 0;
#pragma unroll
  for (int i = 1; i < kMaxSeg; ++i)
    if (i < a.nseg && w_tile >= a.seg_tile0[i]) s = i;
  return s;
}

struct EpiSmem {
  float* rs;     // [TT]   RMS row scale
  float* red;    // [4][16]
  int* redi;     // [4][16]
  float* red2;   // [4][16]
  int* redi2;    // [4][16]
  float* tmx;    // [16]
  float* xch;    // [16][128]
};

// One 16-token chunk of the epilogue for the thread holding weight row fr.
__device__ void epi_chunk(const GemmArgs& a, float (&v)[kEpiTok], int w_tile, int tok0, int rs_off, int fr,
                          int et, int M, const EpiSmem& S) {
  const int q = fr >> 5, lane = fr & 31;
  if (a.ssq_in) {
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) v[j] *= S.rs[rs_off + j];
  }
  if (a.mode == MODE_RESID) {
    const int n = w_tile * kTileN + fr;
    const bool nv = n < a.seg_rows[0];
    const float g = nv ? __bfloat162float(a.g_next[n]) : 0.f;
    float sq[kEpiTok];
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) {
      const int m = tok0 + j;
      float hn = 0.f;
      if (m < M && nv) {
        float* hp = a.h + (size_t)m * a.h_ld + n;
        hn = *hp + v[j];
        *hp = hn;
        __nv_bfloat16 hi, lo;
        split_bf16(hn * g, hi, lo);
        a.x_next[xpk(2 * m, n, a.x_rows)] = hi;
        a.x_next[xpk(2 * m + 1, n, a.x_rows)] = lo;
      }
      sq[j] = hn * hn;
    }
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) {
      const float s = warp_sum(sq[j]);
      if (lane == 0) S.red[q * 16 + j] = s;
    }
    epi_bar();
    if (et < kEpiTok) {
      const int m = tok0 + et;
      if (m < M)
        a.ssq_out[(size_t)w_tile * a.m_cap + m] =
            ((S.red[et] + S.red[16 + et]) + S.red[32 + et]) + S.red[48 + et];
    }
    epi_bar();
  } else if (a.mode == MODE_QKV) {
    const int seg = seg_of(a, w_tile);
    const int n = (w_tile - a.seg_tile0[seg]) * kTileN + fr;
    const bool nv = n < a.seg_rows[seg];
    if (seg < 2) {
#pragma unroll
      for (int j = 0; j < kEpiTok; ++j) S.xch[j * kTileN + fr] = v[j];
      epi_bar();
      const int half = a.hd >> 1, jj = n % a.hd;
      const bool lo_half = jj < half;
      const int pfr = lo_half ? fr + half : fr - half;
      const int fi = lo_half ? jj : jj - half;
#pragma unroll
      for (int j = 0; j < kEpiTok; ++j) {
        const int m = tok0 + j;
        if (m < M) {
          const int pos = a.row_pos[m];
          const float2 cs = a.rope[(size_t)pos * half + fi];
          const float p = S.xch[j * kTileN + pfr];
          v[j] = lo_half ? v[j] * cs.x - p * cs.y : p * cs.y + v[j] * cs.x;
        }
      }
      epi_bar();
    }
    if (nv) {
#pragma unroll
      for (int j = 0; j < kEpiTok; ++j) {
        const int m = tok0 + j;
        if (m >= M) continue;
        if (seg == 0) {
          a.q_out[(size_t)m * a.q_ld + n] = v[j];
        } else {
          const int pos = a.row_pos[m], b = a.row_seq[m];
          if (pos < 0 || pos / a.page_size >= a.pt_ld) { set_status(a.status, ST_BAD_POS); continue; }
          const int page = a.page_table[(size_t)b * a.pt_ld + pos / a.page_size];
          if (page < 0 || page >= a.n_pages) { set_status(a.status, ST_BAD_PAGE); continue; }
          const int kvh = n / a.hd, e = n % a.hd;
          __nv_bfloat16* base = seg == 1 ? a.kcache : a.vcache;
          base[(((size_t)page * a.hkv + kvh) * a.page_size + pos % a.page_size) * a.hd + e] =
              __float2bfloat16_rn(v[j]);
        }
      }
    }
  } else if (a.mode == MODE_SWIGLU) {
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) S.xch[j * kTileN + fr] = v[j];
    epi_bar();
    if (fr < 64) {
      const int n = w_tile * 64 + fr;
      if (n < a.seg_rows[0]) {
#pragma unroll
        for (int j = 0; j < kEpiTok; ++j) {
          const int m = tok0 + j;
          if (m >= M) continue;
          const float gt = S.xch[j * kTileN + fr], up = S.xch[j * kTileN + 64 + fr];
          __nv_bfloat16 hi, lo;
          split_bf16(silu(gt) * up, hi, lo);
          a.x_next[xpk(2 * m, n, a.x_rows)] = hi;
          a.x_next[xpk(2 * m + 1, n, a.x_rows)] = lo;
        }
      }
    }
    epi_bar();
  } else {  // MODE_LOGITS
    const int vi = w_tile * kTileN + fr;
    const bool valid = vi < a.vocab;
    const float T = a.call->temp;
    const bool sample = a.call->sample != 0 && a.row_gi != nullptr;
    float x[kEpiTok];
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) {
      const int m = tok0 + j;
      x[j] = valid ? v[j] : -INFINITY;
      if (a.logits && valid && m < M) {
        const int orow = a.row_out ? a.row_out[m] : m;
        if (orow >= 0) a.logits[(size_t)orow * a.vocab + vi] = v[j];
      }
    }
    // tile max and argmax per row
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) {
      float mv = x[j];
      int mi = valid ? vi : INT_MAX;
      warp_argmax(mv, mi);
      if (lane == 0) { S.red[q * 16 + j] = mv; S.redi[q * 16 + j] = mi; }
    }
    // Gumbel-max draw per row (sampling draft rows only)
    if (sample) {
#pragma unroll 1
      for (int j = 0; j < kEpiTok; ++j) {
        const int m = tok0 + j;
        float gv = -INFINITY;
        int gi = INT_MAX;
        if (m < M && valid) {
          const int ri = a.row_gi[m];
          if (ri >= 0) {
            const uint32_t w = philox_word(a.call->seed, (uint32_t)a.gumbel_stream, a.call->step,
                                           (uint32_t)a.row_seq[m], (uint32_t)ri, (uint32_t)vi);
            gv = x[j] / T + gumbel(w);
            gi = vi;
          }
        }
        warp_argmax(gv, gi);
        if (lane == 0) { S.red2[q * 16 + j] = gv; S.redi2[q * 16 + j] = gi; }
      }
    }
    epi_bar();
    if (et < kEpiTok) {
      float mv = S.red[et];
      int mi = S.redi[et];
      for (int qq = 1; qq < 4; ++qq) argmax_merge(mv, mi, S.red[qq * 16 + et], S.redi[qq * 16 + et]);
      S.tmx[et] = mv;
      S.redi[et] = mi;  // keep the tile argmax
      if (sample) {
        float gv = S.red2[et];
        int gi = S.redi2[et];
        for (int qq = 1; qq < 4; ++qq) argmax_merge(gv, gi, S.red2[qq * 16 + et], S.redi2[qq * 16 + et]);
        S.red2[et] = gv;
        S.redi2[et] = gi;
      }
    }
    epi_bar();
    float e[kEpiTok];
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) e[j] = valid ? expf(x[j] / T - S.tmx[j] / T) : 0.f;
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) {
      const float s = warp_sum(e[j]);
      if (lane == 0) S.red[q * 16 + j] = s;
    }
    epi_bar();
    if (et < kEpiTok) {
      const int m = tok0 + et;
      if (m < M) {
        const float se = ((S.red[et] + S.red[16 + et]) + S.red[32 + et]) + S.red[48 + et];
        const size_t o = (size_t)w_tile * a.m_cap + m;
        a.stats[o] = make_float4(S.tmx[et], se, sample ? S.red2[et] : -INFINITY, 0.f);
        a.stats_i[o] = make_int2(S.redi[et], sample ? S.redi2[et] : -1);
      }
    }
    epi_bar();
  }
}

template <int TT>
__global__ void __launch_bounds__(192, 1) gemm_kernel(const __grid_constant__ GemmArgs a) {
  using C = GemmCfg<TT>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::kStages * C::kABytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + C::kStages * C::kBBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* accf = empty + C::kStages;
  uint64_t* acce = accf + 2;
  uint32_t* misc = reinterpret_cast<uint32_t*>(acce + 2);
  uint32_t* tmem_slot = misc;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 1);
  int* bcast = reinterpret_cast<int*>(misc + 2);
  float* scratch = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(misc) + C::kMiscBytes);
  EpiSmem S;
  S.rs = scratch;
  S.red = S.rs + TT;
  S.redi = reinterpret_cast<int*>(S.red + 64);
  S.red2 = reinterpret_cast<float*>(S.redi + 64);
  S.redi2 = reinterpret_cast<int*>(S.red2 + 64);
  S.tmx = reinterpret_cast<float*>(S.redi2 + 64);
  S.xch = S.tmx + 16;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long U = (long)a.w_tiles * a.tok_tiles * a.kc;
  const long G = gridDim.x;
  const long c = blockIdx.x;
  const long u0 = range_start(c, U, G), u1 = range_start(c + 1, U, G);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(&accf[b], 1); mbar_init(&acce[b], 128); }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      for (int i = 0; i < kMaxSeg; ++i)
        if ((i < a.nseg || (a.pair && i < 2)) && !a.wpk[i]) tma_prefetch_desc(&a.wmap[i]);
      const int n = (int)(u1 - u0);
      const int npre = n < C::kStages ? n : C::kStages;
      // Unit cursor advanced incrementally: the producer issues one stage per
      // wake-up with no divisions on the path between the 'empty' signal and
      // the copies.
      int kk = (int)(u0 % a.kc);
      int w_tile = (int)((u0 / a.kc) / a.tok_tiles), tok_tile = (int)((u0 / a.kc) % a.tok_tiles);
      const __nv_bfloat16* wsrc0 = nullptr;  // packed block base of the current weight tile (A)
      const __nv_bfloat16* wsrc1 = nullptr;  // second half (gate/up pairs)
      const CUtensorMap* wmap0 = nullptr;
      int wrow = 0;                          // row-major fallback: first row of the tile
      auto set_tile = [&]() {
        if (a.pair) {
          if (a.wpk[0]) {
            wsrc0 = a.wpk[0] + (size_t)w_tile * a.kc * 64 * 64;
            wsrc1 = a.wpk[1] + (size_t)w_tile * a.kc * 64 * 64;
          } else {
            wsrc0 = wsrc1 = nullptr;
            wrow = w_tile * 64;
          }
        } else {
          const int seg = seg_of(a, w_tile);
          const int blk = w_tile - a.seg_tile0[seg];
          wsrc0 = a.wpk[seg] ? a.wpk[seg] + (size_t)blk * a.kc * kTileN * 64 : nullptr;
          wmap0 = &a.wmap[seg];
          wrow = blk * kTileN;
        }
      };
      set_tile();
      const size_t x_tile_off = (size_t)2 * TT * 64;      // elements between token tiles of one block
      const size_t x_blk = (size_t)a.x_rows * 64;         // elements between 64-column blocks
      auto issue_a = [&](int s) {
        uint8_t* dst = sA + s * C::kABytes;
        if (a.pair) {
          if (wsrc0) {
            bulk_load_hint(dst, wsrc0 + (size_t)kk * 64 * 64, C::kABytes / 2, &full[s], pol);
            bulk_load_hint(dst + C::kABytes / 2, wsrc1 + (size_t)kk * 64 * 64, C::kABytes / 2, &full[s], pol);
          } else {
            tma_load_2d_hint(dst, &a.wmap[0], &full[s], kk * kChunkK, wrow, pol);
            tma_load_2d_hint(dst + C::kABytes / 2, &a.wmap[1], &full[s], kk * kChunkK, wrow, pol);
          }
        } else if (wsrc0) {
          bulk_load_hint(dst, wsrc0 + (size_t)kk * kTileN * 64, C::kABytes, &full[s], pol);
        } else {
          tma_load_2d_hint(dst, wmap0, &full[s], kk * kChunkK, wrow, pol);
        }
      };
      auto issue_b = [&](int s, int kk_, int tok_) {
        bulk_load(sB + s * C::kBBytes, a.x + (size_t)kk_ * x_blk + (size_t)tok_ * x_tile_off, C::kBBytes, &full[s]);
      };
      auto advance = [&]() {
        if (++kk == a.kc) {
          kk = 0;
          if (++tok_tile == a.tok_tiles) { tok_tile = 0; ++w_tile; }
          set_tile();
        }
      };
      // weights first: they do not depend on the previous kernel
      int pre_kk[C::kStages], pre_tok[C::kStages];
      for (int i = 0; i < npre; ++i) {
        mbar_arrive_expect_tx(&full[i], C::kStageBytes);
        issue_a(i);
        pre_kk[i] = kk;
        pre_tok[i] = tok_tile;
        advance();
      }
      pdl_wait();
      for (int i = 0; i < npre; ++i) issue_b(i, pre_kk[i], pre_tok[i]);
      int s = npre % C::kStages;
      uint32_t ph = (uint32_t)((npre / C::kStages) & 1) ^ 1u;
      for (int i = npre; i < n; ++i) {
        if (!mbar_wait(&empty[s], ph, abort_flag)) {
          set_status(a.status, ST_TIMEOUT_TMA);
          *abort_flag = 1;
          break;
        }
        mbar_arrive_expect_tx(&full[s], C::kStageBytes);
        issue_a(s);
        issue_b(s, kk, tok_tile);
        advance();
        if (++s == C::kStages) { s = 0; ph ^= 1u; }
      }
      pdl_trigger();
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kTileN, 2 * TT);
      long i = 0;
      int seg_i = 0;
      bool ok = true;
      for (long u = u0; u < u1 && ok;) {
        const long t = u / a.kc;
        const long ub = u, ue = (t + 1) * a.kc < u1 ? (t + 1) * a.kc : u1;
        const int ab = seg_i % C::kNumAcc;
        const uint32_t aph = (uint32_t)((seg_i / C::kNumAcc) & 1) ^ 1u;
        if (!mbar_wait(&acce[ab], aph, abort_flag)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d = tmem + ab * C::kAccCols;
        for (; u < ue; ++u, ++i) {
          const int s = (int)(i % C::kStages);
          if (!mbar_wait(&full[s], (uint32_t)((i / C::kStages) & 1), abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint64_t ad = sw128_desc(smem_u32(sA + s * C::kABytes));
          const uint64_t bd = sw128_desc(smem_u32(sB + s * C::kBBytes));
#pragma unroll
          for (int k = 0; k < kChunkK / 16; ++k)
            umma_bf16(d, ad + 2 * k, bd + 2 * k, idesc, (u > ub || k > 0) ? 1u : 0u);
          umma_commit(&empty[s]);
        }
        if (!ok) break;
        umma_commit(&accf[ab]);
        ++seg_i;
      }
      if (!ok) {
        set_status(a.status, ST_TIMEOUT_MMA);
        *abort_flag = 1;
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5) ----------------
    pdl_wait();
    const int et = threadIdx.x - 64;
    const int q = warp & 3;
    const int fr = q * 32 + lane;
    int M = *a.m_dev;
    if (M > a.m_cap) {
      if (et == 0) set_status(a.status, ST_BAD_ROWS);
      M = a.m_cap;
    }
    int seg_i = 0;
    for (long u = u0; u < u1;) {
      const long t = u / a.kc;
      const long ub = u, ue = (t + 1) * a.kc < u1 ? (t + 1) * a.kc : u1;
      u = ue;
      const int ab = seg_i % C::kNumAcc;
      const int w_tile = (int)(t / a.tok_tiles), tok_tile = (int)(t % a.tok_tiles);
      const int tok_base = tok_tile * TT;
      if (a.ssq_in) {
        // all partial sums of squares of this token tile in one round of loads,
        // then a fixed-order sum per row (16 rows at a time through xch)
        for (int c0 = 0; c0 < TT; c0 += kEpiTok) {
          const int nld = a.ssq_tiles * kEpiTok;
          for (int i = et; i < nld; i += 128) {
            const int tile = i / kEpiTok, j = i % kEpiTok;
            const int m = tok_base + c0 + j;
            S.xch[i] = m < M ? __ldcg(a.ssq_in + (size_t)tile * a.m_cap + m) : 0.f;
          }
          epi_bar();
          if (et < kEpiTok) {
            float ss = 0.f;
            for (int t2 = 0; t2 < a.ssq_tiles; ++t2) ss += S.xch[t2 * kEpiTok + et];
            S.rs[c0 + et] = 1.0f / sqrtf(ss * a.inv_d + a.eps);
          }
          epi_bar();
        }
      }
      if (!mbar_wait(&accf[ab], (uint32_t)((seg_i / C::kNumAcc) & 1), abort_flag)) {
        if (et == 0) set_status(a.status, ST_TIMEOUT_EPI);
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      epi_bar();
      const uint32_t tbase = tmem + ab * C::kAccCols + ((uint32_t)(q * 32) << 16);
      const bool whole = (ub == t * a.kc) && (ue == (t + 1) * a.kc);
      if (whole) {
#pragma unroll 1
        for (int ch = 0; ch < C::kChunks; ++ch) {
          uint32_t r[32];
          tmem_ld32(tbase + ch * 32, r);
          float v[kEpiTok];
#pragma unroll
          for (int j = 0; j < kEpiTok; ++j) v[j] = __uint_as_float(r[2 * j]) + __uint_as_float(r[2 * j + 1]);
          epi_chunk(a, v, w_tile, tok_base + ch * kEpiTok, ch * kEpiTok, fr, et, M, S);
        }
      } else {
        const int slot = (ub == u0) ? 0 : 1;
        float* mine = a.partials + ((size_t)c * 2 + slot) * (kTileN * TT);
#pragma unroll 1
        for (int ch = 0; ch < C::kChunks; ++ch) {
          uint32_t r[32];
          tmem_ld32(tbase + ch * 32, r);
          float4* dst = reinterpret_cast<float4*>(mine + ((size_t)ch * kTileN + fr) * kEpiTok);
#pragma unroll
          for (int j4 = 0; j4 < 4; ++j4)
            dst[j4] = make_float4(__uint_as_float(r[8 * j4 + 0]) + __uint_as_float(r[8 * j4 + 1]),
                                  __uint_as_float(r[8 * j4 + 2]) + __uint_as_float(r[8 * j4 + 3]),
                                  __uint_as_float(r[8 * j4 + 4]) + __uint_as_float(r[8 * j4 + 5]),
                                  __uint_as_float(r[8 * j4 + 6]) + __uint_as_float(r[8 * j4 + 7]));
        }
        __threadfence();
        epi_bar();
        const long cf = owner_of(t * a.kc, U, G), cl = owner_of((t + 1) * a.kc - 1, U, G);
        if (et == 0) {
          const int old = atomicAdd(&a.counters[t], 1);
          bcast[0] = (old == (int)(cl - cf)) ? 1 : 0;
        }
        epi_bar();
        if (bcast[0]) {
          __threadfence();
#pragma unroll 1
          for (int ch = 0; ch < C::kChunks; ++ch) {
            uint32_t r[32];
            tmem_ld32(tbase + ch * 32, r);
            float v[kEpiTok];
#pragma unroll
            for (int j = 0; j < kEpiTok; ++j) v[j] = 0.f;
            // contributors in CTA order, four partial tiles requested per round trip
            for (long cc0 = cf; cc0 <= cl; cc0 += 4) {
              float4 pv[4][4];
#pragma unroll
              for (int q4 = 0; q4 < 4; ++q4) {
                const long cc = cc0 + q4;
                if (cc <= cl && cc != c) {
                  const int sl = range_start(cc, U, G) >= t * a.kc ? 0 : 1;
                  const float4* p = reinterpret_cast<const float4*>(
                      a.partials + ((size_t)cc * 2 + sl) * (kTileN * TT) + ((size_t)ch * kTileN + fr) * kEpiTok);
#pragma unroll
                  for (int j4 = 0; j4 < 4; ++j4) pv[q4][j4] = __ldcg(p + j4);
                }
              }
#pragma unroll
              for (int q4 = 0; q4 < 4; ++q4) {
                const long cc = cc0 + q4;
                if (cc > cl) break;
                if (cc == c) {
#pragma unroll
                  for (int j = 0; j < kEpiTok; ++j) v[j] += __uint_as_float(r[2 * j]) + __uint_as_float(r[2 * j + 1]);
                } else {
#pragma unroll
                  for (int j4 = 0; j4 < 4; ++j4) {
                    v[4 * j4 + 0] += pv[q4][j4].x;
                    v[4 * j4 + 1] += pv[q4][j4].y;
                    v[4 * j4 + 2] += pv[q4][j4].z;
                    v[4 * j4 + 3] += pv[q4][j4].w;
                  }
                }
              }
            }
            epi_chunk(a, v, w_tile, tok_base + ch * kEpiTok, ch * kEpiTok, fr, et, M, S);
          }
          if (et == 0) a.counters[t] = 0;
        }
      }
      tc_fence_before();
      mbar_arrive(&acce[ab]);
      epi_bar();
      ++seg_i;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

int gemm_smem_bytes(int tt) {
  switch (tt) {
    case 16: return GemmCfg<16>::kSmem;
    case 32: return GemmCfg<32>::kSmem;
    case 64: return GemmCfg<64>::kSmem;
    default: return -1;
  }
}

template <int TT>
static cudaError_t launch_tt(const GemmArgs& a, int grid, cudaStream_t s, bool pdl) {
  static bool configured = false;
  const int smem = GemmCfg<TT>::kSmem;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(gemm_kernel<TT>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemm_kernel<TT>, a);
}

void launch_gemm(const GemmArgs& a, int tt, int grid, cudaStream_t s, bool pdl) {
  cudaError_t e;
  switch (tt) {
    case 16: e = launch_tt<16>(a, grid, s, pdl); break;
    case 32: e = launch_tt<32>(a, grid, s, pdl); break;
    default: e = launch_tt<64>(a, grid, s, pdl); break;
  }
  if (e != cudaSuccess) throw e;
}

}  // namespace pard
