// Persistent decode pass: one cooperative launch, one CTA per SM, runs every
// phase of a whole forward pass over <= 16 new rows -- per layer the QKV
// GEMM, attention, O GEMM, gate/up GEMM and down GEMM, then the LM head.
//
// Why: at decode sizes each weight-streaming GEMM of a layer moves only
// 33-235 MB, so the start-up latency, split-K fix-up and dependency wait of a
// separate launch per phase cost as much as the streaming itself.  Here the
// producer warp keeps streaming weights across phase boundaries: through a
// 7-stage shared-memory ring, and further ahead as L2 prefetches, so the
// weight tiles of the next phases are in flight while a phase waits for its
// inputs; only the activation tiles of a phase wait for the phase that
// produces them.  Phases signal completion through per-phase counters in
// global memory (release / acquire); every wait is bounded and reports a
// timeout in the status word instead of hanging.
//
// Roles per CTA (192 threads): warp 0 streams (bulk copies), warp 1 issues
// tcgen05.mma into a double-buffered TMEM accumulator, warps 2-5 run the GEMM
// epilogues (shared with the per-phase kernel, gemm_core.cuh) and, in the
// attention phases, the tensor-core attention (attn_core.cuh) with a global
// split combine finished by the last split to arrive.  Each role reads its
// phase description once per phase into registers or shared memory: the
// table lives in global memory, and re-reading it inside the pipelines would
// put an L2 round trip on every step.
#pragma once

#include "attn_core.cuh"
#include "gemm_core.cuh"

namespace pard {

constexpr int kFwdStages = 7;

template <int HD>
struct FwdCfg {
  using Gm = GemmCfg<kFwdTT>;
  static constexpr int kRing = kFwdStages * Gm::kStageBytes;
  static constexpr int kAttnBufs = 3;  // K/V chunk ring (2 chunks in flight)
  static constexpr int kAttn = (AttnCfg<HD, kAttnBufs>::kSmem + 1023) / 1024 * 1024;
  static constexpr int kPhase = (int)((sizeof(Phase) + 127) / 128 * 128);  // epilogue's copy of its phase
  // full, empty, accf x2, acce x2, drain; rounded to 16 bytes so that the
  // epilogue scratch after it takes 16-byte vector accesses
  static constexpr int kBar = (8 * (2 * kFwdStages + 5) + 15) / 16 * 16;
  static constexpr int kMisc = 64;
  static constexpr int kEpiFloats = Gm::kScratchFloats;
  static constexpr int kSmall = (kMaxQV + kMaxQV * kFwdMaxSplit) * 4;
  static constexpr int kSmem = 1024 + kRing + kAttn + kPhase + kBar + kMisc + 4 * kEpiFloats + kSmall + 128;
};

__device__ __forceinline__ bool reached(unsigned v, unsigned target) { return (int)(v - target) >= 0; }

// Phase p complete in every CTA, as seen by a relaxed read (no acquire yet:
// the caller fences once it has seen it, so polling keeps L1 warm).
__device__ __forceinline__ bool phase_seen(const FwdArgs& f, int p) {
  return p < 0 || reached(ld_relaxed_u32(f.done + p), f.target);
}
// Bounded wait for phase p, with acquire semantics on success.
static __device__ bool wait_phase(const FwdArgs& f, int p, volatile int* abort) {
  if (p < 0) return true;
  const unsigned long long t0 = globaltimer();
  while (!phase_seen(f, p)) {
    if (*abort) return false;
    if (globaltimer() - t0 > kWaitLimitNs) return false;
    __nanosleep(32);
  }
  fence_acq_rel_gpu();
  return true;
}

// Work split of a GEMM phase of U (tile, K-chunk) units: the first g =
// min(G, U) CTAs share the units evenly, exactly as a separate launch of g CTAs
// would, so each of them holds at least one unit and the CTAs holding parts of
// one tile are consecutive (the split-K fix-up counts on both); the other CTAs
// hold none.
struct UnitRange {
  long u0, u1, g;
};
__device__ __forceinline__ UnitRange phase_units(long c, long U, long G) {
  const long g = U < G ? U : G;
  return c < g ? UnitRange{range_start(c, U, g), range_start(c + 1, U, g), g} : UnitRange{0, 0, g};
}

// What the producer needs of a GEMM phase, held in registers.
struct ProdPhase {
  const __nv_bfloat16* w[kMaxSeg];  // packed weights per segment
  const __nv_bfloat16* x;           // packed activations
  size_t x_blk;                     // elements between 64-column blocks of x
  int seg1, seg2;                   // first tile of segments 1 and 2
  int nseg, pair, kc, w_tiles, dep;
  __device__ __forceinline__ int seg_of_tile(int t) const {
    return (nseg > 2 && t >= seg2) ? 2 : ((nseg > 1 && t >= seg1) ? 1 : 0);
  }
  __device__ __forceinline__ int seg_first(int seg) const { return seg == 0 ? 0 : (seg == 1 ? seg1 : seg2); }
};
__device__ __forceinline__ ProdPhase load_prod_phase(const Phase& P) {
  ProdPhase q;
  const GemmArgs& a = P.g;
#pragma unroll
  for (int i = 0; i < kMaxSeg; ++i) q.w[i] = a.wpk[i];
  q.x = a.x;
  q.x_blk = (size_t)a.x_rows * 64;
  q.seg1 = a.seg_tile0[1];
  q.seg2 = a.seg_tile0[2];
  q.nseg = a.nseg;
  q.pair = a.pair;
  q.kc = a.kc;
  q.w_tiles = a.w_tiles;
  q.dep = P.dep;
  return q;
}

// L2 prefetch cursor over this CTA's weight units of all GEMM phases, in
// consumption order.  A CTA's units inside one weight segment are one
// contiguous byte range (two for gate/up pairs), so the cursor walks runs of
// units with plain pointer increments.
struct PrefetchCursor {
  const __nv_bfloat16* p0;
  const __nv_bfloat16* p1;  // gate/up pairs: the up half
  uint32_t elems;           // elements per unit per pointer
  long run;                 // units left in the current run
  long u, u1;               // next unit and end of this CTA's range in phase ph
  int ph;                   // phase of the run (n_phases: exhausted)
};

__device__ __forceinline__ void prefetch_next(const FwdArgs& f, long c, long G, PrefetchCursor& q) {
  if (q.run == 0) {
    // next run: the rest of the current segment, else the next phase with units
    while (q.u >= q.u1) {
      if (++q.ph >= f.n_phases) return;
      const Phase& P = f.phases[q.ph];
      if (P.type != PH_GEMM) continue;
      const UnitRange ur = phase_units(c, (long)P.g.w_tiles * P.g.kc, G);
      q.u = ur.u0;
      q.u1 = ur.u1;
    }
    const ProdPhase a = load_prod_phase(f.phases[q.ph]);
    const int t = (int)(q.u / a.kc);
    if (a.pair) {
      q.p0 = a.w[0] + (size_t)q.u * 64 * 64;
      q.p1 = a.w[1] + (size_t)q.u * 64 * 64;
      q.elems = 64 * 64;
      q.run = q.u1 - q.u;
    } else {
      const int seg = a.seg_of_tile(t);
      const long seg_end = seg + 1 < a.nseg ? (long)a.seg_first(seg + 1) * a.kc : (long)a.w_tiles * a.kc;
      q.p0 = a.w[seg] + (size_t)(q.u - (long)a.seg_first(seg) * a.kc) * kTileN * 64;
      q.p1 = nullptr;
      q.elems = kTileN * 64;
      q.run = (q.u1 < seg_end ? q.u1 : seg_end) - q.u;
    }
  }
  bulk_prefetch_l2(q.p0, q.elems * 2);
  q.p0 += q.elems;
  if (q.p1) {
    bulk_prefetch_l2(q.p1, q.elems * 2);
    q.p1 += q.elems;
  }
  --q.run;
  ++q.u;
}

template <int HD, int GROUP>
__global__ void __launch_bounds__(192, 1) fwd_kernel(const __grid_constant__ FwdArgs f) {
  constexpr int TT = kFwdTT, S = kFwdStages;
  using C = GemmCfg<TT>;
  using F = FwdCfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = base;
  uint8_t* sB = sA + S * C::kABytes;
  uint8_t* sAttn = sB + S * C::kBBytes;
  Phase* sPh = reinterpret_cast<Phase*>(sAttn + F::kAttn);
  uint64_t* full = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(sPh) + F::kPhase);
  uint64_t* empty = full + S;
  uint64_t* accf = empty + S;
  uint64_t* acce = accf + 2;
  uint64_t* drain = acce + 2;
  uint32_t* misc = reinterpret_cast<uint32_t*>(reinterpret_cast<uint8_t*>(full) + F::kBar);
  uint32_t* tmem_slot = misc;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 1);
  int* bcast = reinterpret_cast<int*>(misc + 2);
  float* scratch = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(misc) + F::kMisc);
  const EpiSmem Es = carve_epi<TT>(scratch);
  int* s_pos = reinterpret_cast<int*>(scratch + C::kScratchFloats);
  float* s_w = reinterpret_cast<float*>(s_pos + kMaxQV);  // [64][kFwdMaxSplit]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long G = gridDim.x;
  const long c = blockIdx.x;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(&accf[b], 1); mbar_init(&acce[b], 128); }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, 64);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint32_t armed[S];  // producer: times each ring slot was armed
  for (int s = 0; s < S; ++s) armed[s] = 0;
  pdl_wait();     // rows, activations and norms of the embedding kernel
  pdl_trigger();  // dependents start only once every CTA of this grid is running

  if (warp == 0) {
    // ------------------------------ producer ------------------------------
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      int s = 0;
      uint32_t ph = 1;  // parity of the 'empty' phase to wait for (first ring pass is free)
      bool ok = true;
      // L2 prefetch ahead of the ring, across phase boundaries: kFwdPrefetch
      // units while streaming, up to kFwdPrefetchMax while the ring waits for
      // a phase's inputs, so HBM keeps streaming through the dependency waits
      PrefetchCursor pf{nullptr, nullptr, 0, 0, 0, 0, -1};
      int pf_lead = 0;  // units prefetched beyond the ring's issue point
      for (; pf_lead < kFwdPrefetch; ++pf_lead) prefetch_next(f, c, G, pf);
      for (int p = 0; p < f.n_phases && ok; ++p) {
        if (f.phases[p].type != PH_GEMM) continue;
        const ProdPhase a = load_prod_phase(f.phases[p]);
        const UnitRange ur = phase_units(c, (long)a.w_tiles * a.kc, G);
        const int n = (int)(ur.u1 - ur.u0);
        if (n == 0) continue;
        int kk = (int)(ur.u0 % a.kc), w_tile = (int)(ur.u0 / a.kc);
        const __nv_bfloat16 *wsrc0 = nullptr, *wsrc1 = nullptr;
        auto set_tile = [&]() {
          if (a.pair) {
            wsrc0 = a.w[0] + (size_t)w_tile * a.kc * 64 * 64;
            wsrc1 = a.w[1] + (size_t)w_tile * a.kc * 64 * 64;
          } else {
            const int seg = a.seg_of_tile(w_tile);
            wsrc0 = a.w[seg] + (size_t)(w_tile - a.seg_first(seg)) * a.kc * kTileN * 64;
          }
        };
        set_tile();
        // Wait for the phase that produces this phase's activations.  Meanwhile
        // only L2 prefetches go out: data streamed into this SM's shared memory
        // now would queue ahead of the epilogue's stores that finish the
        // producing phase, and the ring refills from L2 once the inputs are in.
        if (!phase_seen(f, a.dep)) {
          const unsigned long long t0 = globaltimer();
          while (!phase_seen(f, a.dep)) {
            for (int j = 0; j < 4 && pf_lead < kFwdPrefetchMax; ++j, ++pf_lead) prefetch_next(f, c, G, pf);
            if (*abort_flag || globaltimer() - t0 > kWaitLimitNs) { ok = false; break; }
          }
          if (!ok) break;
        }
        fence_acq_rel_gpu();
        fence_proxy_async();
        for (int i = 0; i < n && ok; ++i) {
          if (!mbar_wait(&empty[s], ph, abort_flag)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[s], C::kStageBytes);
          ++armed[s];
          uint8_t* dst = sA + s * C::kABytes;
          if (a.pair) {
            bulk_load_hint(dst, wsrc0 + (size_t)kk * 64 * 64, C::kABytes / 2, &full[s], pol);
            bulk_load_hint(dst + C::kABytes / 2, wsrc1 + (size_t)kk * 64 * 64, C::kABytes / 2, &full[s], pol);
          } else {
            bulk_load_hint(dst, wsrc0 + (size_t)kk * kTileN * 64, C::kABytes, &full[s], pol);
          }
          bulk_load(sB + s * C::kBBytes, a.x + (size_t)kk * a.x_blk, C::kBBytes, &full[s]);
          if (--pf_lead < kFwdPrefetch) {
            prefetch_next(f, c, G, pf);
            ++pf_lead;
          }
          if (++kk == a.kc) {
            kk = 0;
            ++w_tile;
            set_tile();
          }
          if (++s == S) { s = 0; ph ^= 1u; }
        }
      }
      if (!ok) {
        set_status(f.status, ST_TIMEOUT_TMA);
        *abort_flag = 1;
      }
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer ------------------------------
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kTileN, 2 * TT);
      long i = 0;
      int seg_i = 0;
      bool ok = true;
      for (int p = 0; p < f.n_phases && ok; ++p) {
        if (f.phases[p].type != PH_GEMM) continue;
        const long kc = f.phases[p].g.kc;
        const long U = (long)f.phases[p].g.w_tiles * kc;
        const UnitRange ur = phase_units(c, U, G);
        const long u0 = ur.u0, u1 = ur.u1;
        for (long u = u0; u < u1 && ok;) {
          const long t = u / kc;
          const long ub = u, ue = (t + 1) * kc < u1 ? (t + 1) * kc : u1;
          const int ab = seg_i & 1;
          if (!mbar_wait(&acce[ab], (uint32_t)((seg_i >> 1) & 1) ^ 1u, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t d = tmem + ab * C::kAccCols;
          for (; u < ue; ++u, ++i) {
            const int s = (int)(i % S);
            if (!mbar_wait(&full[s], (uint32_t)((i / S) & 1), abort_flag)) { ok = false; break; }
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
      }
      if (!ok) {
        set_status(f.status, ST_TIMEOUT_MMA);
        *abort_flag = 1;
      }
    }
  } else {
    // --------------------- epilogues and attention (warps 2..5) ---------------------
    const int et = threadIdx.x - 64;
    const int q = warp & 3;
    const int fr = q * 32 + lane;
    int M = *f.m_dev;
    if (M > f.m_cap) {
      if (et == 0) set_status(f.status, ST_BAD_ROWS);
      M = f.m_cap;
    }
    int seg_i = 0;
    bool ok = true;
    for (int p = 0; p < f.n_phases && ok; ++p) {
      // this phase's description into shared memory, and (one thread) the
      // acquire of the phase whose outputs it reads
      {
        const uint4* src = reinterpret_cast<const uint4*>(f.phases + p);
        uint4* dst = reinterpret_cast<uint4*>(sPh);
        for (int i = et; i < (int)(sizeof(Phase) / 16); i += 128) dst[i] = src[i];
      }
      if (et == 0) {
        const int dep = f.phases[p].dep;
        if (!wait_phase(f, dep, abort_flag)) {
          set_status(f.status, ST_TIMEOUT_EPI);
          *abort_flag = 1;
        }
      }
      if (epi_bar_any(*abort_flag != 0)) break;
      const Phase& P = *sPh;
      if (P.type == PH_GEMM) {
        const GemmArgs& a = P.g;
        const long kc = a.kc;
        const long U = (long)a.w_tiles * kc;
        const UnitRange ur = phase_units(c, U, G);
        const long u0 = ur.u0, u1 = ur.u1;
        for (long u = u0; u < u1;) {
          const long t = u / kc;
          const long ub = u, ue = (t + 1) * kc < u1 ? (t + 1) * kc : u1;
          u = ue;
          const int ab = seg_i & 1;
          if (!mbar_wait(&accf[ab], (uint32_t)((seg_i >> 1) & 1), abort_flag)) {
            if (et == 0) set_status(f.status, ST_TIMEOUT_EPI);
            *abort_flag = 1;
            ok = false;
          }
          if (epi_bar_any(*abort_flag != 0)) { ok = false; break; }
          tc_fence_after();
          if (a.ssq_in) epi_row_scale<TT>(a, 0, et, M, Es);  // sums of squares of the previous phase
          const uint32_t tbase = tmem + ab * C::kAccCols + ((uint32_t)(q * 32) << 16);
          epi_segment<TT>(a, t, ub, ue, u0, U, ur.g, c, tbase, (int)t, 0, fr, et, M, Es, bcast);
          tc_fence_before();
          mbar_arrive(&acce[ab]);
          epi_bar();
          ++seg_i;
        }
        if (!ok) break;
      } else {
        // attention items of this CTA: (group, split) = c, c + G, ...
        const AttnArgs& at = P.at;
        const int ns = P.attn_split;
        const int items = P.attn_groups * ns;
        for (int it = (int)c; it < items; it += (int)G) {
          const int gidx = it / ns, sp = it % ns;
          const int rb = gidx % at.row_blocks;
          const int kvh = (gidx / at.row_blocks) % at.hkv;
          const int b = gidx / (at.row_blocks * at.hkv);
          const AttnRows R = attn_unit<HD, GROUP, F::kAttnBufs>(at, b, kvh, rb, sp, ns, M, sAttn, s_pos, et,
                                                                [] { epi_bar(); }, [] {});
          const int row0 = R.row0, nqv = R.nrows * GROUP;
          epi_bar();  // every warp's partial is in shared memory
          const float* part = reinterpret_cast<const float*>(sAttn);
          if (ns == 1) {
            for (int i = et; i < nqv * (HD / 4); i += 128) {
              const int qv = i / (HD / 4), d4 = i % (HD / 4);
              const float* src = part + qv * AttnCfg<HD, F::kAttnBufs>::kPartLd;
              const float inv = 1.0f / src[HD + 1];
              const float4 v = make_float4(src[4 * d4] * inv, src[4 * d4 + 1] * inv, src[4 * d4 + 2] * inv,
                                           src[4 * d4 + 3] * inv);
              store_pair4(at.x_out, row0 + qv / GROUP, (kvh * GROUP + qv % GROUP) * HD + 4 * d4, at.x_rows, v);
            }
            epi_bar();
            continue;
          }
          // this split's partial in global memory: o as [split][64][HD] rows
          // (16-byte aligned), then (m, l) as [split][64] pairs
          float* go = f.attn_part + (size_t)gidx * ns * kMaxQV * (HD + 2);
          float2* gml = reinterpret_cast<float2*>(go + (size_t)ns * kMaxQV * HD);
          for (int i = et; i < nqv * (HD / 4); i += 128) {
            const int qv = i / (HD / 4), d4 = i % (HD / 4);
            const float* src = part + qv * AttnCfg<HD, F::kAttnBufs>::kPartLd + 4 * d4;
            reinterpret_cast<float4*>(go + ((size_t)sp * kMaxQV + qv) * HD)[d4] =
                make_float4(src[0], src[1], src[2], src[3]);
          }
          for (int qv = et; qv < nqv; qv += 128)
            gml[sp * kMaxQV + qv] = make_float2(part[qv * AttnCfg<HD, F::kAttnBufs>::kPartLd + HD],
                                                 part[qv * AttnCfg<HD, F::kAttnBufs>::kPartLd + HD + 1]);
          epi_bar();
          if (et == 0) {
            const int old = atom_add_acq_rel(&f.attn_cnt[gidx], 1);  // publishes ours, acquires the others'
            bcast[0] = old == ns - 1 ? 1 : 0;
          }
          epi_bar();
          if (bcast[0]) {
            // combine the splits in split order; every split's loads in flight at once
            for (int qv = et; qv < nqv; qv += 128) {
              float2 ml[kFwdMaxSplit];
#pragma unroll
              for (int r = 0; r < kFwdMaxSplit; ++r)
                ml[r] = r < ns ? __ldcg(gml + r * kMaxQV + qv) : make_float2(-INFINITY, 0.f);
              float mx = -INFINITY;
#pragma unroll
              for (int r = 0; r < kFwdMaxSplit; ++r) mx = fmaxf(mx, ml[r].x);
              float w[kFwdMaxSplit], L = 0.f;
#pragma unroll
              for (int r = 0; r < kFwdMaxSplit; ++r) {
                w[r] = ml[r].x == -INFINITY ? 0.f : expf(ml[r].x - mx);
                L += ml[r].y * w[r];
              }
#pragma unroll
              for (int r = 0; r < kFwdMaxSplit; ++r) s_w[qv * kFwdMaxSplit + r] = w[r] / L;
            }
            epi_bar();
            // two outputs per thread per round: 2 x ns loads in flight
            const int n_out = nqv * (HD / 4);
            for (int i0 = et; i0 < n_out; i0 += 256) {
              float4 pv[2][kFwdMaxSplit];
#pragma unroll
              for (int u = 0; u < 2; ++u) {
                const int i = i0 + u * 128;
                const int qv = i / (HD / 4), d4 = i % (HD / 4);
#pragma unroll
                for (int r = 0; r < kFwdMaxSplit; ++r)
                  pv[u][r] = (i < n_out && r < ns)
                                 ? __ldcg(reinterpret_cast<const float4*>(go + ((size_t)r * kMaxQV + qv) * HD) + d4)
                                 : make_float4(0.f, 0.f, 0.f, 0.f);
              }
#pragma unroll
              for (int u = 0; u < 2; ++u) {
                const int i = i0 + u * 128;
                if (i >= n_out) break;
                const int qv = i / (HD / 4), d4 = i % (HD / 4);
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int r = 0; r < kFwdMaxSplit; ++r) {
                  const float wr = r < ns ? s_w[qv * kFwdMaxSplit + r] : 0.f;
                  if (wr != 0.f) {
                    acc.x += pv[u][r].x * wr;
                    acc.y += pv[u][r].y * wr;
                    acc.z += pv[u][r].z * wr;
                    acc.w += pv[u][r].w * wr;
                  }
                }
                store_pair4(at.x_out, row0 + qv / GROUP, (kvh * GROUP + qv % GROUP) * HD + 4 * d4, at.x_rows, acc);
              }
            }
            if (et == 0) f.attn_cnt[gidx] = 0;
          }
          epi_bar();
        }
      }
      // this CTA's share of phase p is complete (all stores, fix-ups,
      // combines): the barrier orders every thread's stores before the one
      // release (cumulative) that publishes them
      fence_proxy_async();
      epi_bar();
      if (et == 0) red_release_add(f.done + p, 1u);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // let this CTA's copies and MMAs in flight land before its memory goes away
    if (warp == 0 && lane == 0)
      for (int s = 0; s < S; ++s)
        if (armed[s]) mbar_drain(&full[s], (armed[s] - 1) & 1u);
    if (warp == 1 && lane == 0) {
      umma_commit(drain);
      mbar_drain(drain, 0);
    }
    __syncthreads();
  }
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 64);
  }
}

template <int HD, int GROUP>
cudaError_t launch_fwd_t(const FwdArgs& f, int grid, cudaStream_t s) {
  static bool configured = false;
  const int smem = FwdCfg<HD>::kSmem;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(fwd_kernel<HD, GROUP>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;  // every CTA resident at once (they wait on each other)
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  cudaError_t e = cudaLaunchKernelEx(&cfg, fwd_kernel<HD, GROUP>, f);
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    cfg.numAttrs = 1;  // without programmatic serialization
    e = cudaLaunchKernelEx(&cfg, fwd_kernel<HD, GROUP>, f);
  }
  return e;
}

// one translation unit per head size (fwd_hd128.cu, fwd_hd64.cu)
cudaError_t launch_fwd_hd128(const FwdArgs& f, int group, int grid, cudaStream_t s);
cudaError_t launch_fwd_hd64(const FwdArgs& f, int group, int grid, cudaStream_t s);

}  // namespace pard
