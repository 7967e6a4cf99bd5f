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
//    CTAs; a tile shared by several CTAs is finished by the first of them,
//    for which it is the last segment: the others store their partials and
//    signal with one release increment each, the finisher pulls all partials
//    into its idle stage ring with bulk copies and sums them in CTA order
//    (deterministic);
//  * epilogues are fused: RMS row scaling, RoPE + paged KV write (QKV),
//    residual add + next norm's gain and sum of squares (O / down),
//    SiLU(gate) * up (gate/up pairs), logits + per-tile max / argmax /
//    sum-exp / Gumbel-max statistics (LM head);
//  * programmatic dependent launch: the weight tiles of the first stages
//    are requested before waiting on the previous kernel, since weights do
//    not depend on it.
#include "gemm_core.cuh"

namespace pard {

template <int TT>
// two CTAs per SM at the 16-token tile: this launch's and the next one's
__global__ void __launch_bounds__(192, TT <= 16 ? 2 : 1) gemm_kernel(const __grid_constant__ GemmArgs a) {
  using C = GemmCfg<TT>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::kStages * C::kABytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + C::kStages * C::kBBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* accf = empty + C::kStages;
  uint64_t* acce = accf + 2;
  uint64_t* drain = acce + 2;
  uint64_t* fx = drain + 1;  // split-K finish: partials pulled into the ring
  // the barrier block is rounded to 16 bytes: the epilogue scratch after
  // misc takes 16-byte vector accesses
  uint32_t* misc = reinterpret_cast<uint32_t*>(reinterpret_cast<uint8_t*>(full) + C::kBarBytes);
  static_assert(C::kStages * C::kStageBytes % 16 == 0 && C::kBarBytes % 16 == 0 && C::kMiscBytes % 16 == 0 &&
                    TT % 4 == 0,
                "epilogue scratch alignment");
  uint32_t* tmem_slot = misc;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 1);
  int* bcast = reinterpret_cast<int*>(misc + 2);
  volatile int* fx_armed = reinterpret_cast<volatile int*>(misc + 3);
  float* scratch = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(misc) + C::kMiscBytes);
  const EpiSmem S = carve_epi<TT>(scratch);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int* live = reinterpret_cast<int*>(misc + 4);  // [0] token tiles processed, [1] token rows of one tile's MMA
  // this CTA's units (recomputed below in the rare launch that drops token tiles)
  const bool early = a.m_early && a.tok_tiles > 1;
  const long G = gridDim.x;
  const long c = blockIdx.x;
  long U = (long)a.w_tiles * a.tok_tiles * a.kc;
  long u0 = range_start(c, U, G), u1 = range_start(c + 1, U, G);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(&accf[b], 1); mbar_init(&acce[b], 128); }
    mbar_init(drain, 1);
    mbar_init(fx, 1);
    *abort_flag = 0;
    *fx_armed = 0;
    // Token tiles past the pass's row count hold no output row.  A
    // multi-tile launch whose row count was written two or more launches back
    // (the previous kernel itself waited for that writer before letting this
    // grid start) reads it now and neither loads nor multiplies those tiles;
    // when one tile is left it covers only the rows present (B = 2 n_tok
    // rows).  A single-tile launch takes n_tok from the host's row capacity
    // and starts without this read.
    if (early) {
      const int m = min(max(__ldcg(a.m_dev), 1), a.m_cap);
      const int tiles = min(a.tok_tiles, (m + TT - 1) / TT);
      live[0] = tiles;
      live[1] = tiles == 1 ? min(TT, (m + 7) / 8 * 8) : TT;
    }
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int tok_tiles = early ? live[0] : a.tok_tiles;
  if (tok_tiles != a.tok_tiles) {
    U = (long)a.w_tiles * tok_tiles * a.kc;
    u0 = range_start(c, U, G);
    u1 = range_start(c + 1, U, G);
  }
  uint32_t armed[C::kStages];  // producer: times each ring slot was armed
  for (int s = 0; s < C::kStages; ++s) armed[s] = 0;
  // ring slots this launch uses, and how many are filled before the PDL wait
  const int R = (a.stages > 0 && a.stages < C::kStages) ? a.stages : C::kStages;
  const int P = (a.pre_stages > 0 && a.pre_stages < R) ? a.pre_stages : R;
  // token rows a tile's MMA covers: hi/lo pairs are the B rows, so N = 2 n_tok
  const int n_tok = early ? live[1]
                           : ((a.tok_tiles == 1 && a.n_tok > 0 && a.n_tok < TT && a.n_tok % 8 == 0) ? a.n_tok : TT);
  const uint32_t b_bytes = (uint32_t)n_tok * 2 * 128;
  const uint32_t stage_bytes = (uint32_t)C::kABytes + b_bytes;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      for (int i = 0; i < kMaxSeg; ++i)
        if ((i < a.nseg || (a.pair && i < 2)) && !a.wpk[i]) tma_prefetch_desc(&a.wmap[i]);
      const int n = (int)(u1 - u0);
      const int npre = n < P ? n : P;
      // Unit cursor advanced incrementally: the producer issues one stage per
      // wake-up with no divisions on the path between the 'empty' signal and
      // the copies.
      int kk = (int)(u0 % a.kc);
      int w_tile = (int)((u0 / a.kc) / tok_tiles), tok_tile = (int)((u0 / a.kc) % tok_tiles);
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
        bulk_load(sB + s * C::kBBytes, a.x + (size_t)kk_ * x_blk + (size_t)tok_ * x_tile_off, b_bytes, &full[s]);
      };
      auto advance = [&]() {
        if (++kk == a.kc) {
          kk = 0;
          if (++tok_tile == tok_tiles) { tok_tile = 0; ++w_tile; }
          set_tile();
        }
      };
      // weights first: they do not depend on the previous kernel
      int pre_kk[C::kStages], pre_tok[C::kStages];
      for (int i = 0; i < npre; ++i) {
        mbar_arrive_expect_tx(&full[i], stage_bytes);
        ++armed[i];
        issue_a(i);
        pre_kk[i] = kk;
        pre_tok[i] = tok_tile;
        advance();
      }
      pdl_wait();
      for (int i = 0; i < npre; ++i) issue_b(i, pre_kk[i], pre_tok[i]);
      int s = npre % R;
      uint32_t ph = (uint32_t)((npre / R) & 1) ^ 1u;
      for (int i = npre; i < n; ++i) {
        if (!mbar_wait(&empty[s], ph, abort_flag)) {
          set_status(a.status, ST_TIMEOUT_TMA);
          *abort_flag = 1;
          break;
        }
        mbar_arrive_expect_tx(&full[s], stage_bytes);
        ++armed[s];
        issue_a(s);
        issue_b(s, kk, tok_tile);
        advance();
        if (++s == R) { s = 0; ph ^= 1u; }
      }
      pdl_trigger();
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kTileN, 2 * n_tok);
      int s = 0;          // ring slot of the next unit
      uint32_t fph = 0;   // its 'full' phase parity
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
        for (; u < ue; ++u) {
          if (!mbar_wait(&full[s], fph, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint64_t ad = sw128_desc(smem_u32(sA + s * C::kABytes));
          const uint64_t bd = sw128_desc(smem_u32(sB + s * C::kBBytes));
#pragma unroll
          for (int k = 0; k < kChunkK / 16; ++k)
            umma_bf16(d, ad + 2 * k, bd + 2 * k, idesc, (u > ub || k > 0) ? 1u : 0u);
          umma_commit(&empty[s]);
          if (++s == R) { s = 0; fph ^= 1u; }
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
    int rs_tok = -1;  // token tile whose RMS row scale S.rs holds
    for (long u = u0; u < u1;) {
      const long t = u / a.kc;
      const long ub = u, ue = (t + 1) * a.kc < u1 ? (t + 1) * a.kc : u1;
      u = ue;
      const int ab = seg_i % C::kNumAcc;
      const int w_tile = (int)(t / tok_tiles), tok_tile = (int)(t % tok_tiles);
      const int tok_base = tok_tile * TT;
      if (a.ssq_in && tok_base != rs_tok) {
        epi_row_scale<TT>(a, tok_base, et, M, S);
        rs_tok = tok_base;
      }
      // result-independent loads of a segment this CTA finishes (it starts
      // the tile), issued while the MMAs run
      EpiPre pre0 = {};
      if (ub == t * a.kc) pre0 = epi_pre(a, w_tile, tok_base, et, M);
      if (!mbar_wait(&accf[ab], (uint32_t)((seg_i / C::kNumAcc) & 1), abort_flag)) {
        if (et == 0) set_status(a.status, ST_TIMEOUT_EPI);
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      epi_bar();
      const uint32_t tbase = tmem + ab * C::kAccCols + ((uint32_t)(q * 32) << 16);
      if (!epi_segment_owned<TT>(a, t, ub, ue, u0, U, G, c, tbase, w_tile, tok_base, fr, et, M, S, pre0,
                                 reinterpret_cast<float*>(sA), (uint32_t)(C::kStages * C::kStageBytes), fx,
                                 fx_armed, abort_flag, bcast))
        break;
      tc_fence_before();
      mbar_arrive(&acce[ab]);
      epi_bar();
      ++seg_i;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // let this CTA's copies and MMAs in flight land before its memory goes away
    if (warp == 0 && lane == 0)
      for (int s = 0; s < C::kStages; ++s)
        if (armed[s]) mbar_drain(&full[s], (armed[s] - 1) & 1u);
    if (warp == 1 && lane == 0) {
      umma_commit(drain);
      mbar_drain(drain, 0);
    }
    // fx_armed: 1 + the staging round whose copies may be in flight
    if (threadIdx.x == 64 && *fx_armed) mbar_drain(fx, (uint32_t)((*fx_armed - 1) & 1));
    __syncthreads();
  }
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

int gemm_smem_bytes(int tt) {
  switch (tt) {
    case 16: return GemmCfg<16>::kSmem;
    case 64: return GemmCfg<64>::kSmem;
    case 128: return GemmCfg<128>::kSmem;
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
    case 64: e = launch_tt<64>(a, grid, s, pdl); break;
    default: e = launch_tt<128>(a, grid, s, pdl); break;
  }
  if (e != cudaSuccess) throw e;
}

}  // namespace pard
