// Device code of the weight-streaming GEMM (gemm.cu): tile configuration,
// the fused epilogues and the split-K finish.
#pragma once

#include <climits>

#include "common.cuh"
#include "internal.h"

namespace pard {

template <int TT>
struct GemmCfg {
  static constexpr int kABytes = kTileN * 128;       // 128 rows x 64 bf16
  static constexpr int kBBytes = 2 * TT * 128;       // 2*TT rows x 64 bf16
  static constexpr int kStageBytes = kABytes + kBBytes;
  // Ring capacity (a launch may use fewer).  At the 16-token tile the CTA
  // (about 106 KB of shared memory, at most 168 registers a thread) leaves
  // room on its SM for one CTA of the next launch, which then starts, fills
  // its ring and reaches its PDL wait while this one finishes.  Wider tiles
  // run one CTA per SM and take a deeper ring (~200 KB) instead: with 4 and
  // 3 stages they kept too few weight bytes in flight per SM.  The 128-token
  // tile (65-128 rows: one pass over the weights for all of them) fits 4
  // stages of 48 KB.
  static constexpr int kStages = TT <= 16 ? 5 : (TT <= 32 ? 8 : (TT <= 64 ? 6 : 4));
  static constexpr int kAccCols = 2 * TT;
  static constexpr int kNumAcc = (2 * kAccCols <= 512) ? 2 : 1;
  static constexpr int kTmemCols = kNumAcc * kAccCols <= 32 ? 32 : kNumAcc * kAccCols <= 64 ? 64
                                   : kNumAcc * kAccCols <= 128 ? 128 : kNumAcc * kAccCols <= 256 ? 256 : 512;
  static constexpr int kChunks = TT / kEpiTok;
  // scratch after the stage ring
  // full, empty, accf x2, acce x2, drain, fix-up; rounded to 16 bytes
  static constexpr int kBarBytes = (8 * (2 * kStages + 6) + 15) / 16 * 16;
  static constexpr int kMiscBytes = 64;
  static constexpr int kScratchFloats = TT + kEpiTok * kTileN + 3 * kEpiTok;
  static constexpr int kSmem = 1024 + kStages * kStageBytes + kBarBytes + kMiscBytes + 4 * kScratchFloats;
};

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }
// epi_bar that also returns whether any of the 128 threads passed v != 0, so
// that all of them take the same branch after it
__device__ __forceinline__ bool epi_bar_any(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, 1, 128, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)v)
      : "memory");
  return r != 0;
}

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
  float* xch;    // [16][128] the chunk's accumulator, exchanged to row-major (16-byte aligned)
  int* ri;       // [3][16] per-row facts of the chunk, loaded once by 16 threads
};

// Carves the epilogue scratch (GemmCfg<TT>::kScratchFloats floats) at p.
template <int TT>
__device__ __forceinline__ EpiSmem carve_epi(float* p) {
  EpiSmem S;
  S.rs = p;
  S.xch = S.rs + TT;
  S.ri = reinterpret_cast<int*>(S.xch + kEpiTok * kTileN);
  return S;
}

// Eight consecutive columns (col % 8 == 0) of activation row m as bf16 hi/lo
// pairs in the packed layout: one 16-byte chunk in each of rows 2m and 2m+1.
__device__ __forceinline__ void store_pair8(__nv_bfloat16* x, int m, int col, int x_rows, const float (&v)[8]) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    __nv_bfloat16 h0, l0, h1, l1;
    split_bf16(v[2 * e], h0, l0);
    split_bf16(v[2 * e + 1], h1, l1);
    h[e] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
    l[e] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
  }
  *reinterpret_cast<uint4*>(x + xpk(2 * m, col, x_rows)) = make_uint4(h[0], h[1], h[2], h[3]);
  *reinterpret_cast<uint4*>(x + xpk(2 * m + 1, col, x_rows)) = make_uint4(l[0], l[1], l[2], l[3]);
}

// Loads of one 16-token chunk's epilogue that do not depend on the tile's
// result: the residual and norm gains (O / down), the row's position, KV page
// and RoPE factors (QKV), the rows' output facts (LM head).  Taken before the
// split-K arrival, so that the CTA that finishes a tile has them in hand.
struct EpiPre {
  uint4 w[8];     // O / down: h (w[0..3] as float4) and g (w[4..5]); QKV: 16 (cos, sin) pairs
  int pos, page;  // QKV: position (-1 invalid) and KV page (-1 none) of the thread's token
  int ri[3];      // LM head, threads et < 16: logits row, Gumbel index, sequence of token et
  int ok;         // O / down: the vector loads above were taken
};

static __device__ __forceinline__ EpiPre epi_pre(const GemmArgs& a, int w_tile, int tok0, int et, int M) {
  EpiPre p;
  p.ok = 0;
  p.pos = -1;
  p.page = -1;
  const int jl = et >> 3, c16 = (et & 7) * 16;
  const int mr = tok0 + jl;
  if (a.mode == MODE_RESID) {
    const int n0 = w_tile * kTileN + c16;
    if (mr < M && n0 + 16 <= a.seg_rows[0] && (reinterpret_cast<uintptr_t>(a.g_next) & 15) == 0) {
      // L2 loads: h was written by the previous kernel's CTAs
      const float4* hp = reinterpret_cast<const float4*>(a.h + (size_t)mr * a.h_ld + n0);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float4 h = __ldcg(hp + i);
        p.w[i] = make_uint4(__float_as_uint(h.x), __float_as_uint(h.y), __float_as_uint(h.z), __float_as_uint(h.w));
      }
#pragma unroll
      for (int i = 0; i < 2; ++i) p.w[4 + i] = *reinterpret_cast<const uint4*>(a.g_next + n0 + 8 * i);
      p.ok = 1;
    }
  } else if (a.mode == MODE_QKV) {
    const int seg = seg_of(a, w_tile);
    const int n0 = (w_tile - a.seg_tile0[seg]) * kTileN + c16;
    if (mr < M) {
      const int pos = a.row_pos[mr];
      const bool pv = pos >= 0 && pos / a.page_size < a.pt_ld;
      if (!pv && (et & 7) == 0) set_status(a.status, ST_BAD_POS);
      if (pv) {
        p.pos = pos;
        if (seg > 0) {
          const int page = a.page_table[(size_t)a.row_seq[mr] * a.pt_ld + pos / a.page_size];
          if (page >= 0 && page < a.n_pages) p.page = page;
          else if ((et & 7) == 0) set_status(a.status, ST_BAD_PAGE);
        }
        if (seg < 2 && n0 < a.seg_rows[seg]) {
          const int half = a.hd >> 1, jj = n0 % a.hd;
          const int fi0 = jj < half ? jj : jj - half;
          const uint4* csp = reinterpret_cast<const uint4*>(a.rope + (size_t)pos * half + fi0);
#pragma unroll
          for (int i = 0; i < 8; ++i) p.w[i] = csp[i];
        }
      }
    }
  } else if (a.mode == MODE_LOGITS) {
    if (et < kEpiTok) {
      const int m = tok0 + et;
      const bool in = m < M;
      const bool sample = a.call->sample != 0 && a.row_gi != nullptr;
      p.ri[0] = in ? (a.row_out ? a.row_out[m] : m) : -1;
      p.ri[1] = (in && sample) ? a.row_gi[m] : -1;
      p.ri[2] = (in && sample) ? a.row_seq[m] : 0;
    }
  }
  return p;
}

// One 16-token chunk of the epilogue for the thread holding weight row fr;
// pre holds the chunk's result-independent loads (epi_pre).
static __device__ void epi_chunk(const GemmArgs& a, float (&v)[kEpiTok], int w_tile, int tok0, int rs_off, int fr,
                          int et, int M, const EpiSmem& S, const EpiPre& pre) {
  if (a.ssq_in) {
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) v[j] *= S.rs[rs_off + j];
  }
  // Row-major phase: after the accumulator columns are exchanged through
  // S.xch, thread et handles token jl = et / 8 and the 16 consecutive tile rows
  // (output columns) c16 .. c16+15, c16 = 16 (et % 8), so the stores are
  // 16-byte vectors instead of one scalar per token.
  const int jl = et >> 3, c16 = (et & 7) * 16;
  const int mr = tok0 + jl;  // this thread's token in the row-major phase
  if (a.mode == MODE_RESID) {
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) S.xch[j * kTileN + fr] = v[j];
    epi_bar();
    const int n0 = w_tile * kTileN + c16;
    float sq = 0.f;
    if (mr < M && n0 < a.seg_rows[0]) {
      const float* xv = S.xch + jl * kTileN + c16;
      float* hp = a.h + (size_t)mr * a.h_ld + n0;
      if (pre.ok) {
        float4 hv[4];
        uint4 gv[2];
#pragma unroll
        for (int i = 0; i < 4; ++i)
          hv[i] = make_float4(__uint_as_float(pre.w[i].x), __uint_as_float(pre.w[i].y), __uint_as_float(pre.w[i].z),
                              __uint_as_float(pre.w[i].w));
#pragma unroll
        for (int i = 0; i < 2; ++i) gv[i] = pre.w[4 + i];
        float hn[16];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float4 x4 = reinterpret_cast<const float4*>(xv)[i];  // xv: 16-float aligned
          hn[4 * i + 0] = hv[i].x + x4.x;
          hn[4 * i + 1] = hv[i].y + x4.y;
          hn[4 * i + 2] = hv[i].z + x4.z;
          hn[4 * i + 3] = hv[i].w + x4.w;
          reinterpret_cast<float4*>(hp)[i] = make_float4(hn[4 * i], hn[4 * i + 1], hn[4 * i + 2], hn[4 * i + 3]);
        }
        const __nv_bfloat16* gb = reinterpret_cast<const __nv_bfloat16*>(gv);
#pragma unroll
        for (int h8 = 0; h8 < 2; ++h8) {
          float o[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) o[e] = hn[8 * h8 + e] * __bfloat162float(gb[8 * h8 + e]);
          store_pair8(a.x_next, mr, n0 + 8 * h8, a.x_rows, o);
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) sq += hn[i] * hn[i];
      } else {
        for (int i = 0; i < 16 && n0 + i < a.seg_rows[0]; ++i) {
          const float hn = __ldcg(hp + i) + xv[i];
          hp[i] = hn;
          __nv_bfloat16 hi, lo;
          split_bf16(hn * __bfloat162float(a.g_next[n0 + i]), hi, lo);
          a.x_next[xpk(2 * mr, n0 + i, a.x_rows)] = hi;
          a.x_next[xpk(2 * mr + 1, n0 + i, a.x_rows)] = lo;
          sq += hn * hn;
        }
      }
    }
    // the tile's sum of squares of this token: its 8 threads are 8 adjacent lanes
    sq += __shfl_xor_sync(0xffffffffu, sq, 1);
    sq += __shfl_xor_sync(0xffffffffu, sq, 2);
    sq += __shfl_xor_sync(0xffffffffu, sq, 4);
    if ((et & 7) == 0 && mr < M) a.ssq_out[(size_t)w_tile * a.m_cap + mr] = sq;
    epi_bar();  // S.xch is rewritten by the next chunk
  } else if (a.mode == MODE_QKV) {
    const int seg = seg_of(a, w_tile);
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) S.xch[j * kTileN + fr] = v[j];
    epi_bar();
    const int n0 = (w_tile - a.seg_tile0[seg]) * kTileN + c16;  // first column within the segment
    const int pos = pre.pos;
    if (mr < M && n0 < a.seg_rows[seg] && pos >= 0) {
      const float* xv = S.xch + jl * kTileN;
      float o[16];
#pragma unroll
      for (int i4 = 0; i4 < 4; ++i4) {
        const float4 x4 = reinterpret_cast<const float4*>(xv + c16)[i4];
        o[4 * i4] = x4.x; o[4 * i4 + 1] = x4.y; o[4 * i4 + 2] = x4.z; o[4 * i4 + 3] = x4.w;
      }
      if (seg < 2) {
        // rotate-half RoPE: the 16 columns lie in one half of one head, and the
        // partner half of that head is in the same 128-row tile
        const int half = a.hd >> 1, jj = n0 % a.hd;
        const bool lo_half = jj < half;
        const int pc = lo_half ? c16 + half : c16 - half;
        float4 cs4[8];  // 16 (cos, sin) pairs
#pragma unroll
        for (int i = 0; i < 8; ++i)
          cs4[i] = make_float4(__uint_as_float(pre.w[i].x), __uint_as_float(pre.w[i].y), __uint_as_float(pre.w[i].z),
                               __uint_as_float(pre.w[i].w));
        float pr[16];  // the partner half (pc: a multiple of 16 columns)
#pragma unroll
        for (int i4 = 0; i4 < 4; ++i4) {
          const float4 x4 = reinterpret_cast<const float4*>(xv + pc)[i4];
          pr[4 * i4] = x4.x; pr[4 * i4 + 1] = x4.y; pr[4 * i4 + 2] = x4.z; pr[4 * i4 + 3] = x4.w;
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float c = (i & 1) ? cs4[i >> 1].z : cs4[i >> 1].x;
          const float sn = (i & 1) ? cs4[i >> 1].w : cs4[i >> 1].y;
          const float p = pr[i];
          o[i] = lo_half ? o[i] * c - p * sn : p * sn + o[i] * c;
        }
      }
      if (seg == 0) {
        float4* qp = reinterpret_cast<float4*>(a.q_out + (size_t)mr * a.q_ld + n0);
#pragma unroll
        for (int i = 0; i < 4; ++i) qp[i] = make_float4(o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
      } else {
        const int page = pre.page;
        if (page >= 0) {
          const int kvh = n0 / a.hd, e0 = n0 % a.hd;
          __nv_bfloat16* base = seg == 1 ? a.kcache : a.vcache;
          __nv_bfloat16* dst =
              base + (((size_t)page * a.hkv + kvh) * a.page_size + pos % a.page_size) * a.hd + e0;
          uint32_t w[8];
#pragma unroll
          for (int i = 0; i < 8; ++i)
            w[i] = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(o[2 * i])) |
                   ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(o[2 * i + 1])) << 16);
          reinterpret_cast<uint4*>(dst)[0] = make_uint4(w[0], w[1], w[2], w[3]);
          reinterpret_cast<uint4*>(dst)[1] = make_uint4(w[4], w[5], w[6], w[7]);
        }
      }
    }
    epi_bar();  // S.xch is rewritten by the next chunk
  } else if (a.mode == MODE_SWIGLU) {
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) S.xch[j * kTileN + fr] = v[j];
    epi_bar();
    // thread et: token et / 8, output columns 8 (et % 8) .. +8 of the tile's
    // 64 (gate rows 0..63 and up rows 64..127 of the exchange); one 16-byte
    // store per hi / lo row instead of 16 scalar ones
    {
      const int jl = et >> 3, c8 = (et & 7) * 8;
      const int m = tok0 + jl, n0 = w_tile * 64 + c8;
      if (m < M && n0 < a.seg_rows[0]) {
        const float* gp = S.xch + jl * kTileN + c8;
        float out[8];
        const float4 g0 = reinterpret_cast<const float4*>(gp)[0], g1 = reinterpret_cast<const float4*>(gp)[1];
        const float4 u0 = reinterpret_cast<const float4*>(gp + 64)[0], u1 = reinterpret_cast<const float4*>(gp + 64)[1];
        out[0] = silu(g0.x) * u0.x; out[1] = silu(g0.y) * u0.y; out[2] = silu(g0.z) * u0.z; out[3] = silu(g0.w) * u0.w;
        out[4] = silu(g1.x) * u1.x; out[5] = silu(g1.y) * u1.y; out[6] = silu(g1.z) * u1.z; out[7] = silu(g1.w) * u1.w;
        if (n0 + 8 <= a.seg_rows[0]) {
          store_pair8(a.x_next, m, n0, a.x_rows, out);
        } else {
          for (int e = 0; e < 8 && n0 + e < a.seg_rows[0]; ++e) {
            __nv_bfloat16 hi, lo;
            split_bf16(out[e], hi, lo);
            a.x_next[xpk(2 * m, n0 + e, a.x_rows)] = hi;
            a.x_next[xpk(2 * m + 1, n0 + e, a.x_rows)] = lo;
          }
        }
      }
    }
    epi_bar();
  } else {  // MODE_LOGITS
    const float T = a.call->temp;
    const bool sample = a.call->sample != 0 && a.row_gi != nullptr;
    // row facts of the chunk: logits row (-1: none), Gumbel index (-1: none), sequence
    if (et < kEpiTok) {
      S.ri[et] = pre.ri[0];
      S.ri[kEpiTok + et] = pre.ri[1];
      S.ri[2 * kEpiTok + et] = pre.ri[2];
    }
#pragma unroll
    for (int j = 0; j < kEpiTok; ++j) S.xch[j * kTileN + fr] = v[j];
    epi_bar();
    // Row-major phase: thread et reduces token jl's 16 vocabulary entries
    // c16 .. c16 + 15 of the tile in registers, then merges with the other 7
    // threads of its token (adjacent lanes) by three shuffles.
    const int m = tok0 + jl;
    const int n0 = w_tile * kTileN + c16;
    float x[16];
    {
      const float4* xr = reinterpret_cast<const float4*>(S.xch + jl * kTileN + c16);
#pragma unroll
      for (int i4 = 0; i4 < 4; ++i4) {
        const float4 q4 = xr[i4];
        x[4 * i4 + 0] = q4.x; x[4 * i4 + 1] = q4.y; x[4 * i4 + 2] = q4.z; x[4 * i4 + 3] = q4.w;
      }
    }
    const int orow = S.ri[jl];
    if (a.logits && orow >= 0 && m < M) {
      float* lp = a.logits + (size_t)orow * a.vocab + n0;
      if (n0 + 16 <= a.vocab && (a.vocab & 3) == 0) {
#pragma unroll
        for (int i4 = 0; i4 < 4; ++i4)
          reinterpret_cast<float4*>(lp)[i4] = make_float4(x[4 * i4], x[4 * i4 + 1], x[4 * i4 + 2], x[4 * i4 + 3]);
      } else {
        for (int i = 0; i < 16 && n0 + i < a.vocab; ++i) lp[i] = x[i];
      }
    }
    // tile max and argmax (lowest index on ties) of token jl
    float mv = -INFINITY;
    int mi = INT_MAX;
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (n0 + i < a.vocab) argmax_merge(mv, mi, x[i], n0 + i);
#pragma unroll
    for (int o = 4; o > 0; o >>= 1) {
      const float v2 = __shfl_xor_sync(0xffffffffu, mv, o);
      const int i2 = __shfl_xor_sync(0xffffffffu, mi, o);
      argmax_merge(mv, mi, v2, i2);
    }
    // sum of exp((x - max) / T) over the tile
    float se = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i) se += (n0 + i < a.vocab) ? expf(x[i] / T - mv / T) : 0.f;
    se += __shfl_xor_sync(0xffffffffu, se, 4);
    se += __shfl_xor_sync(0xffffffffu, se, 2);
    se += __shfl_xor_sync(0xffffffffu, se, 1);
    // Gumbel-max draw of the tile (sampling draft rows only)
    float gv = -INFINITY;
    int gi = INT_MAX;
    if (sample) {
      const int ri = S.ri[kEpiTok + jl];
      if (m < M && ri >= 0) {
        const uint32_t sq = (uint32_t)S.ri[2 * kEpiTok + jl];
        for (int i = 0; i < 16; ++i)
          if (n0 + i < a.vocab)
            argmax_merge(gv, gi, gumbel_score(x[i], T, a.call->seed, (uint32_t)a.gumbel_stream, a.call->step, sq,
                                              (uint32_t)ri, (uint32_t)(n0 + i)),
                         n0 + i);
      }
#pragma unroll
      for (int o = 4; o > 0; o >>= 1) {
        const float v2 = __shfl_xor_sync(0xffffffffu, gv, o);
        const int i2 = __shfl_xor_sync(0xffffffffu, gi, o);
        argmax_merge(gv, gi, v2, i2);
      }
    }
    if ((et & 7) == 0 && m < M) {
      const size_t o = (size_t)w_tile * a.m_cap + m;
      a.stats[o] = make_float4(mv, se, sample ? gv : -INFINITY, 0.f);
      a.stats_i[o] = make_int2(mi, sample ? gi : -1);
    }
    epi_bar();  // S.xch and the row facts are rewritten by the next chunk
  }
}


// Bounded wait until every bit of `all` is set in *p, with acquire semantics
// on success.
__device__ __forceinline__ bool wait_mask(const unsigned long long* p, unsigned long long all, volatile int* abort) {
  if ((ld_acquire_u64(p) & all) == all) return true;
  const unsigned long long t0 = globaltimer();
  while (true) {
    if ((ld_acquire_u64(p) & all) == all) return true;
    if (*abort) return false;
    if (globaltimer() - t0 > kWaitLimitNs) return false;
  }
}
// bits of contributors 1..n of a tile (bit k - 1: the k-th after the finisher)
__device__ __forceinline__ unsigned long long contrib_bits(int n) { return n >= 64 ? ~0ull : ((1ull << n) - 1); }
// 4-token groups of a 16-token chunk that hold some of the pass's M rows: a
// partial tile stores and copies only those ([chunk][j4][row] layout)
__device__ __forceinline__ int chunk_groups(int M, int tok0) { return min(4, max(0, (M - tok0 + 3) / 4)); }

// Split-K with a designated finisher (per-phase kernel).  The first CTA of a
// tile in CTA order, cf, finishes it.  Its share of the tile is the last
// segment of its range (the tile starts inside the range and runs past its
// end), so when its epilogue gets there every MMA of the CTA has completed and
// the stage ring is idle.  The other contributors move on without a round
// trip: contributor k (the k-th CTA after cf) stores its partial and sets
// bit k - 1 of the tile's arrival mask with one release OR; cf copies each
// partial into the ring as soon as its bit is seen (so the copies of early
// contributors overlap the wait for late ones) and adds them to its own in
// CTA order (deterministic).  With many chunks
// (wide tiles) the copies go in rounds of chunks once every bit is set.
// pre0: epi_pre of the segment's first chunk, taken by the caller before the
// accumulator was ready; only read for a whole tile or by cf.
// ring/ring_bytes: the stage ring; fx: an mbarrier whose phase r is round r
// of the one split tile a CTA finishes; fx_armed: 1 + the round whose copies
// may be in flight (0: none).  Partials hold only the 4-token groups with
// output rows (chunk_groups).  The arrival masks live in a.counters (64-bit
// words, tile t at word t; the host keeps every tile's contributors at 64 or
// fewer) and are cleared by the finisher.
template <int TT>
__device__ bool epi_segment_owned(const GemmArgs& a, long t, long ub, long ue, long u0, long U, long G, long c,
                                  uint32_t tbase, int w_tile, int tok_base, int fr, int et, int M, const EpiSmem& S,
                                  const EpiPre& pre0, float* ring, uint32_t ring_bytes, uint64_t* fx,
                                  volatile int* fx_armed, volatile int* abort_flag, int* bcast) {
  using C = GemmCfg<TT>;
  constexpr int kTileF = kTileN * TT;  // floats of one partial tile
  // 16-token chunks holding at least one of the pass's M rows; the others are
  // neither finished nor exchanged (their rows are not outputs)
  const int nch = max(0, min(C::kChunks, (M - tok_base + kEpiTok - 1) / kEpiTok));
  const int kChF = kTileN * kEpiTok;   // floats of one chunk of a partial tile
  if (ub == t * a.kc && ue == (t + 1) * a.kc) {
    EpiPre pre = pre0;  // one chunk's loads live at a time
#pragma unroll 1
    for (int ch = 0; ch < nch; ++ch) {
      if (ch > 0) pre = epi_pre(a, w_tile, tok_base + ch * kEpiTok, et, M);
      uint32_t r[32];
      tmem_ld32(tbase + ch * 32, r);
      float v[kEpiTok];
#pragma unroll
      for (int j = 0; j < kEpiTok; ++j) v[j] = __uint_as_float(r[2 * j]) + __uint_as_float(r[2 * j + 1]);
      epi_chunk(a, v, w_tile, tok_base + ch * kEpiTok, ch * kEpiTok, fr, et, M, S, pre);
    }
    return true;
  }
  const long cf = owner_of(t * a.kc, U, G), cl = owner_of((t + 1) * a.kc - 1, U, G);
  unsigned long long* mask = reinterpret_cast<unsigned long long*>(a.counters) + t;
  if (c != cf) {
    const int slot = (ub == u0) ? 0 : 1;
    float* mine = a.partials + ((size_t)c * 2 + slot) * kTileF;
#pragma unroll 1
    for (int ch = 0; ch < nch; ++ch) {
      uint32_t r[32];
      tmem_ld32(tbase + ch * 32, r);
      const int ng = chunk_groups(M, tok_base + ch * kEpiTok);
      // [chunk][j4][row] float4s: a warp's accesses are 512 contiguous bytes
      float4* dst = reinterpret_cast<float4*>(mine + (size_t)ch * kTileN * kEpiTok) + fr;
#pragma unroll
      for (int j4 = 0; j4 < 4; ++j4)
        if (j4 < ng)
          dst[j4 * kTileN] = make_float4(__uint_as_float(r[8 * j4 + 0]) + __uint_as_float(r[8 * j4 + 1]),
                                __uint_as_float(r[8 * j4 + 2]) + __uint_as_float(r[8 * j4 + 3]),
                                __uint_as_float(r[8 * j4 + 4]) + __uint_as_float(r[8 * j4 + 5]),
                                __uint_as_float(r[8 * j4 + 6]) + __uint_as_float(r[8 * j4 + 7]));
    }
    // the barrier orders every thread's partial before the one release OR
    // (cumulative)
    epi_bar();
    if (et == 0) red_release_or64(mask, 1ull << (c - cf - 1));
    return true;
  }
  if constexpr (C::kChunks == 1) {
    // 16-token tile: one chunk, so one staging round (the partials of up to
    // ring_bytes / 8 KB contributors) or direct loads
    const int n_other = (int)(cl - cf);
    // bytes copied of one contributor: the 4-token groups of its chunk with output rows
    const uint32_t part_bytes = nch > 0 ? (uint32_t)chunk_groups(M, tok_base) * kTileN * 16 : 0u;
    const bool staged = nch > 0 && (uint32_t)n_other * kChF * 4 <= ring_bytes;
    if (et == 0) {
      const unsigned long long all = contrib_bits(n_other);
      bool ok = true;
      if (staged) {
        *fx_armed = 1;
        mbar_arrive_expect_tx(fx, (uint32_t)n_other * part_bytes);
        // copy each contributor's partial as soon as its bit is seen
        unsigned long long seen = 0;
        const unsigned long long t0 = globaltimer();
        while (seen != all) {
          const unsigned long long m = ld_acquire_u64(mask) & all;
          unsigned long long nw = m & ~seen;
          if (nw) {
            // the partials were written through the generic proxy; the copies
            // read them through the async proxy
            fence_proxy_async();
            while (nw) {
              const int k = __ffsll((long long)nw) - 1;
              nw &= nw - 1;
              const long cc = cf + 1 + k;
              const int sl = range_start(cc, U, G) >= t * a.kc ? 0 : 1;
              bulk_load(ring + (size_t)k * kChF, a.partials + ((size_t)cc * 2 + sl) * kTileF, part_bytes, fx);
            }
            seen = m;
          } else if (*abort_flag || globaltimer() - t0 > kWaitLimitNs) {
            ok = false;
            break;
          }
        }
      } else {
        ok = wait_mask(mask, all, abort_flag);
      }
      if (!ok) set_status(a.status, ST_TIMEOUT_EPI);
      bcast[0] = ok ? 1 : 0;
    }
    epi_bar();
    if (!bcast[0]) {
      *abort_flag = 1;
      return false;
    }
    const bool late = staged && nch > 0 && !mbar_wait(fx, 0, abort_flag);
    if (epi_bar_any(late)) {
      if (et == 0) set_status(a.status, ST_TIMEOUT_EPI);
      *abort_flag = 1;
      return false;
    }
    EpiPre pre = pre0;
  #pragma unroll 1
    for (int ch = 0; ch < nch; ++ch) {
      if (ch > 0) pre = epi_pre(a, w_tile, tok_base + ch * kEpiTok, et, M);
      uint32_t r[32];
      tmem_ld32(tbase + ch * 32, r);
      float v[kEpiTok];
  #pragma unroll
      for (int j = 0; j < kEpiTok; ++j) v[j] = __uint_as_float(r[2 * j]) + __uint_as_float(r[2 * j + 1]);
      const size_t off = (size_t)ch * kTileN * kEpiTok;
      for (int k = 0; k < n_other; ++k) {
        float4 pv[4];
        if (staged) {
          const float4* p = reinterpret_cast<const float4*>(ring + (size_t)k * kChF + off) + fr;
  #pragma unroll
          for (int j4 = 0; j4 < 4; ++j4) pv[j4] = p[j4 * kTileN];
        } else {
          const long cc = cf + 1 + k;
          const int sl = range_start(cc, U, G) >= t * a.kc ? 0 : 1;
          const float4* p = reinterpret_cast<const float4*>(a.partials + ((size_t)cc * 2 + sl) * kTileF + off) + fr;
  #pragma unroll
          for (int j4 = 0; j4 < 4; ++j4) pv[j4] = __ldcg(p + j4 * kTileN);
        }
  #pragma unroll
        for (int j4 = 0; j4 < 4; ++j4) {
          v[4 * j4 + 0] += pv[j4].x;
          v[4 * j4 + 1] += pv[j4].y;
          v[4 * j4 + 2] += pv[j4].z;
          v[4 * j4 + 3] += pv[j4].w;
        }
      }
      epi_chunk(a, v, w_tile, tok_base + ch * kEpiTok, ch * kEpiTok, fr, et, M, S, pre);
    }
  } else {
    const int n_other = (int)(cl - cf);
    // Partials are staged in the idle ring in rounds of chunks: each round one
    // bulk copy per contributor brings the same run of chunks of every
    // partial ([chunk][j4][row] layout: a run of chunks is contiguous), so a
    // tile with many contributors or many chunks costs a few round trips
    // instead of one L2 load chain per chunk.
    const uint32_t ch_bytes = (uint32_t)kChF * 4;
    int per_round = n_other > 0 ? (int)(ring_bytes / ((uint32_t)n_other * ch_bytes)) : nch;
    if (per_round > nch) per_round = nch;
    const bool staged = per_round > 0 && nch > 0;
    if (et == 0) {
      const bool ok = wait_mask(mask, contrib_bits(n_other), abort_flag);
      if (!ok) set_status(a.status, ST_TIMEOUT_EPI);
      bcast[0] = ok ? 1 : 0;
    }
    epi_bar();
    if (!bcast[0]) {
      *abort_flag = 1;
      return false;
    }
    EpiPre pre = pre0;
    const int step = staged ? per_round : nch;
    for (int r0 = 0, round = 0; r0 < nch; r0 += step, ++round) {
      const int r1 = min(nch, r0 + step), nr = r1 - r0;
      if (staged) {
        if (et == 0) {
          // the partials were written through the generic proxy (and the ring
          // read through it by the previous round); the copies use the async proxy
          fence_proxy_async();
          *fx_armed = round + 1;
          mbar_arrive_expect_tx(fx, (uint32_t)n_other * nr * ch_bytes);
          for (int k = 0; k < n_other; ++k) {
            const long cc = cf + 1 + k;
            const int sl = range_start(cc, U, G) >= t * a.kc ? 0 : 1;
            bulk_load(ring + (size_t)k * nr * kChF, a.partials + ((size_t)cc * 2 + sl) * kTileF + (size_t)r0 * kChF,
                      (uint32_t)nr * ch_bytes, fx);
          }
        }
        const bool late = !mbar_wait(fx, (uint32_t)(round & 1), abort_flag);
        if (epi_bar_any(late)) {
          if (et == 0) set_status(a.status, ST_TIMEOUT_EPI);
          *abort_flag = 1;
          return false;
        }
      }
  #pragma unroll 1
      for (int ch = r0; ch < r1; ++ch) {
        if (ch > 0) pre = epi_pre(a, w_tile, tok_base + ch * kEpiTok, et, M);
        uint32_t r[32];
        tmem_ld32(tbase + ch * 32, r);
        float v[kEpiTok];
  #pragma unroll
        for (int j = 0; j < kEpiTok; ++j) v[j] = __uint_as_float(r[2 * j]) + __uint_as_float(r[2 * j + 1]);
        for (int k = 0; k < n_other; ++k) {
          float4 pv[4];
          if (staged) {
            const float4* p = reinterpret_cast<const float4*>(ring + ((size_t)k * nr + (ch - r0)) * kChF) + fr;
  #pragma unroll
            for (int j4 = 0; j4 < 4; ++j4) pv[j4] = p[j4 * kTileN];
          } else {
            const long cc = cf + 1 + k;
            const int sl = range_start(cc, U, G) >= t * a.kc ? 0 : 1;
            const float4* p = reinterpret_cast<const float4*>(a.partials + ((size_t)cc * 2 + sl) * kTileF +
                                                              (size_t)ch * kChF) + fr;
  #pragma unroll
            for (int j4 = 0; j4 < 4; ++j4) pv[j4] = __ldcg(p + j4 * kTileN);
          }
  #pragma unroll
          for (int j4 = 0; j4 < 4; ++j4) {
            v[4 * j4 + 0] += pv[j4].x;
            v[4 * j4 + 1] += pv[j4].y;
            v[4 * j4 + 2] += pv[j4].z;
            v[4 * j4 + 3] += pv[j4].w;
          }
        }
        epi_chunk(a, v, w_tile, tok_base + ch * kEpiTok, ch * kEpiTok, fr, et, M, S, pre);
      }
      if (staged && r1 < nch) epi_bar();  // the ring is read out before the next round's copies
    }
  }
  if (et == 0) *mask = 0ull;
  return true;
}

// RMS row scale for the token tile starting at tok_base: all partial sums of
// squares in one round of loads, then a fixed-order sum per row.
template <int TT>
__device__ void epi_row_scale(const GemmArgs& a, int tok_base, int et, int M, const EpiSmem& S) {
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

}  // namespace pard
