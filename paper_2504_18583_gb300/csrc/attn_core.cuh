// Shared device code of the paged multi-query-position GQA attention: the
// per-(sequence, kv head, row block) partial over a range of 32-key chunks on
// the tensor cores.  Included by the cluster attention kernel (attention.cu).
#pragma once

#include <cuda_fp16.h>

#include "common.cuh"
#include "internal.h"

namespace pard {

constexpr int kAttnThreads = 128;  // 4 warps x 16 query vectors
constexpr int kMaxQV = kMaxQVRows;
constexpr int kKeyChunk = 32;
constexpr int kMaxCluster = kMaxAttnSplit;  // key splits of one work unit (clusters above 8 are non-portable)
constexpr int kAttnPageCache = 512;  // page ids of one work unit's key range held in shared memory

// Shared memory of one work unit: NBUF K/V chunk buffers (a ring, NBUF - 1
// chunks in flight), Q as fp16 rows (the MMA A operand, read with ldmatrix),
// then the page id cache; the partial result (o, m, l) reuses the front at the
// end.
template <int HD, int NBUF>
struct AttnCfg {
  static constexpr int kRowBytes = HD * 2 + 16;             // padded smem row (conflict-free ldmatrix)
  static constexpr int kTileBytes = kKeyChunk * kRowBytes;  // one K or V chunk
  static constexpr int kKV = NBUF * 2 * kTileBytes;         // K and V chunk ring
  static constexpr int kQBytes = kMaxQV * kRowBytes;        // Q rows
  static constexpr int kQOff = kKV;
  static constexpr int kPartLd = HD + 4;                     // partial row: o[HD], m, l, 2 pad (16-byte rows)
  static constexpr int kPart = kMaxQV * kPartLd * 4;        // partial (o, m, l) per CTA
  static constexpr int kPageOff = (kKV + kQBytes) > kPart ? (kKV + kQBytes) : kPart;
  static constexpr int kSmem = kPageOff + kAttnPageCache * 4 + 256;
};

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// register-only (not volatile): the compiler may interleave independent MMAs
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// two fp32 -> fp16x2 (lower-index element in the low half)
__device__ __forceinline__ uint32_t pack_h2(float x0, float x1) {
  const __half2 h = __floats2half2_rn(x0, x1);
  return *reinterpret_cast<const uint32_t*>(&h);
}
// bf16x2 -> fp16x2; exact for magnitudes in [2^-14, 65504] (fp16 keeps more
// significand bits than bf16), rounded below, infinite above
__device__ __forceinline__ uint32_t bf2_to_h2(uint32_t x) {
  return pack_h2(__uint_as_float(x << 16), __uint_as_float(x & 0xffff0000u));
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2_trans(uint32_t& r0, uint32_t& r1, uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];" : "=r"(r0), "=r"(r1) : "r"(addr));
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_size() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// two consecutive floats (8-byte aligned) of CTA `rank`'s shared memory
__device__ __forceinline__ float2 ld_dsmem2(const float* local, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  float2 v;
  asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(remote) : "memory");
  return v;
}

// Four consecutive columns (col % 4 == 0) of activation row m as bf16 hi/lo
// pairs in the packed layout: 8 contiguous bytes in each of rows 2m and 2m+1.
__device__ __forceinline__ void store_pair4(__nv_bfloat16* x, int m, int col, int x_rows, float4 v) {
  __nv_bfloat16 h[4], l[4];
  split_bf16(v.x, h[0], l[0]);
  split_bf16(v.y, h[1], l[1]);
  split_bf16(v.z, h[2], l[2]);
  split_bf16(v.w, h[3], l[3]);
  uint2 hv, lv;
  hv.x = (uint32_t)__bfloat16_as_ushort(h[0]) | ((uint32_t)__bfloat16_as_ushort(h[1]) << 16);
  hv.y = (uint32_t)__bfloat16_as_ushort(h[2]) | ((uint32_t)__bfloat16_as_ushort(h[3]) << 16);
  lv.x = (uint32_t)__bfloat16_as_ushort(l[0]) | ((uint32_t)__bfloat16_as_ushort(l[1]) << 16);
  lv.y = (uint32_t)__bfloat16_as_ushort(l[2]) | ((uint32_t)__bfloat16_as_ushort(l[3]) << 16);
  *reinterpret_cast<uint2*>(x + xpk(2 * m, col, x_rows)) = hv;
  *reinterpret_cast<uint2*>(x + xpk(2 * m + 1, col, x_rows)) = lv;
}

// ---- cluster barrier halves, distributed shared memory bulk copies --------
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive() { asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory"); }
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }
// shared::cluster address of the same offset in CTA `rank`'s shared memory
__device__ __forceinline__ uint32_t mapa_shared(const void* local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(local)), "r"(rank));
  return r;
}
// bytes (multiple of 16, both ends 16-byte aligned) of this CTA's shared
// memory into a peer's, completion counted on the peer's mbarrier
__device__ __forceinline__ void bulk_copy_to_peer(uint32_t dst_cluster, const void* src, uint32_t bytes,
                                                  uint32_t mbar_cluster) {
  asm volatile(
      "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst_cluster),
      "r"(smem_u32(src)), "r"(bytes), "r"(mbar_cluster)
      : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// this thread's bulk copies have finished reading their sources
__device__ __forceinline__ void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// orders this thread's generic-proxy shared memory writes before its async-proxy reads
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// K and V rows of one 32-key chunk into shared memory; positions past maxpos
// (masked anyway) and bad pages become zeros.  spg: the sequence's page table
// row in shared memory (nullptr: read it from global memory here).
template <int HD, int NBUF>
__device__ __forceinline__ void load_chunk(const AttnArgs& a, const int* pt, const int* spg, int kvh, int chunk,
                                           int maxpos, uint8_t* sK, uint8_t* sV, int tid) {
  using C = AttnCfg<HD, NBUF>;
  constexpr int kCh = HD * 2 / 16;
  for (int i = tid; i < kKeyChunk * kCh; i += kAttnThreads) {
    const int key = i / kCh, ch = i % kCh;
    const int pos = chunk * kKeyChunk + key;
    uint8_t* dk = sK + key * C::kRowBytes + ch * 16;
    uint8_t* dv = sV + key * C::kRowBytes + ch * 16;
    int page = -1;
    if (pos <= maxpos && pos / a.page_size < a.pt_ld) {
      page = spg ? spg[pos / a.page_size] : pt[pos / a.page_size];
      if (page < 0 || page >= a.n_pages) {
        set_status(a.status, ST_BAD_PAGE);
        page = -1;
      }
    }
    if (page < 0) {
      *reinterpret_cast<uint4*>(dk) = make_uint4(0, 0, 0, 0);
      *reinterpret_cast<uint4*>(dv) = make_uint4(0, 0, 0, 0);
      continue;
    }
    const size_t off = (((size_t)page * a.hkv + kvh) * a.page_size + pos % a.page_size) * HD + ch * 8;
    cp_async16(dk, a.kcache + off);
    cp_async16(dv, a.vcache + off);
  }
}

// The same thread's pieces of a landed chunk (load_chunk's mapping), bf16 ->
// fp16 in place; zero-filled pieces are zeros in both formats.
template <int HD, int NBUF>
__device__ __forceinline__ void chunk_to_f16(uint8_t* sK, uint8_t* sV, int tid) {
  using C = AttnCfg<HD, NBUF>;
  constexpr int kCh = HD * 2 / 16;
  for (int i = tid; i < kKeyChunk * kCh; i += kAttnThreads) {
    const int key = i / kCh, ch = i % kCh;
    uint4* pk = reinterpret_cast<uint4*>(sK + key * C::kRowBytes + ch * 16);
    uint4* pv = reinterpret_cast<uint4*>(sV + key * C::kRowBytes + ch * 16);
    const uint4 k = *pk, v = *pv;
    *pk = make_uint4(bf2_to_h2(k.x), bf2_to_h2(k.y), bf2_to_h2(k.z), bf2_to_h2(k.w));
    *pv = make_uint4(bf2_to_h2(v.x), bf2_to_h2(v.y), bf2_to_h2(v.z), bf2_to_h2(v.w));
  }
}

// Wait until at most n of this thread's most recent cp.async groups are pending.
__device__ __forceinline__ void cp_async_wait_upto(int n) {
  if (n <= 0) asm volatile("cp.async.wait_group 0;" ::: "memory");
  else if (n == 1) asm volatile("cp.async.wait_group 1;" ::: "memory");
  else asm volatile("cp.async.wait_group 2;" ::: "memory");
}

struct AttnRows {
  int row0, nrows;
  int n_chunks;  // 32-key chunks of the unit's key range (all splits)
};

// A unit whose query vectors fit in two warps and which walks at least this
// many chunks splits every chunk's keys between two warp pairs (see attn_unit).
constexpr int kKeyHalvesMinChunks = 3;

// Online-softmax attention of one warp's 16 query vectors (rows qa = 16 q +
// g and qb = qa + 8 of the lane's quad g) over keys koff .. koff + 8 NJG - 1
// of the chunk ch landed in sK / sV (fp16): S = Q K^T on NJG 8-key n-tiles,
// scale and causal mask (key position <= row position), running max / sum
// update with the rescale of o, then O += P V with P as the A fragments.
template <int HD, int NJG, int ROWB>
__device__ __forceinline__ void attn_chunk(const uint8_t* sK, const uint8_t* sV, int koff, int ch, uint32_t q_base,
                                           int posa, int posb, float scale, float (&o)[HD / 8][4], float& ma,
                                           float& mb, float& la, float& lb, int lane) {
  constexpr int KS = HD / 16;
  constexpr int NT = HD / 8;
  const int g = lane >> 2, c4 = lane & 3;
  // NACC accumulator sets over alternate k-steps keep four independent MMA
  // chains in flight when the warp covers only NJG = 2 n-tiles
  constexpr int NACC = NJG >= 4 ? 1 : 4 / NJG;
  float sacc[NACC][NJG][4];
#pragma unroll
  for (int r = 0; r < NACC; ++r)
#pragma unroll
    for (int j = 0; j < NJG; ++j) sacc[r][j][0] = sacc[r][j][1] = sacc[r][j][2] = sacc[r][j][3] = 0.f;
#pragma unroll
  for (int ks = 0; ks < KS; ++ks) {
    uint32_t qf[4], kb[NJG][2];
    ldsm_x4(qf, q_base + ks * 32);
#pragma unroll
    for (int j = 0; j < NJG; ++j) {
      const uint8_t* krow = sK + (koff + j * 8 + g) * ROWB;
      kb[j][0] = *reinterpret_cast<const uint32_t*>(krow + (ks * 16 + 2 * c4) * 2);
      kb[j][1] = *reinterpret_cast<const uint32_t*>(krow + (ks * 16 + 8 + 2 * c4) * 2);
    }
    // independent accumulators back to back
#pragma unroll
    for (int j = 0; j < NJG; ++j) mma_f16_16816(sacc[ks % NACC][j], qf, kb[j][0], kb[j][1]);
  }
  float s[NJG][4];
#pragma unroll
  for (int j = 0; j < NJG; ++j)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      float v = sacc[0][j][e];
#pragma unroll
      for (int r = 1; r < NACC; ++r) v += sacc[r][j][e];
      s[j][e] = v;
    }
  // scale, causal mask, online softmax (rows qa and qb)
  float mxa = -INFINITY, mxb = -INFINITY;
#pragma unroll
  for (int j = 0; j < NJG; ++j) {
    const int kp = ch * kKeyChunk + koff + j * 8 + 2 * c4;
    s[j][0] = kp <= posa ? s[j][0] * scale : -INFINITY;
    s[j][1] = kp + 1 <= posa ? s[j][1] * scale : -INFINITY;
    s[j][2] = kp <= posb ? s[j][2] * scale : -INFINITY;
    s[j][3] = kp + 1 <= posb ? s[j][3] * scale : -INFINITY;
    mxa = fmaxf(mxa, fmaxf(s[j][0], s[j][1]));
    mxb = fmaxf(mxb, fmaxf(s[j][2], s[j][3]));
  }
  mxa = fmaxf(mxa, __shfl_xor_sync(0xffffffffu, mxa, 1));
  mxa = fmaxf(mxa, __shfl_xor_sync(0xffffffffu, mxa, 2));
  mxb = fmaxf(mxb, __shfl_xor_sync(0xffffffffu, mxb, 1));
  mxb = fmaxf(mxb, __shfl_xor_sync(0xffffffffu, mxb, 2));
  const float mna = fmaxf(ma, mxa), mnb = fmaxf(mb, mxb);
  const float ca = mna == -INFINITY ? 1.f : expf(ma - mna);
  const float cb = mnb == -INFINITY ? 1.f : expf(mb - mnb);
  float sa = 0.f, sb = 0.f;
#pragma unroll
  for (int j = 0; j < NJG; ++j) {
    s[j][0] = s[j][0] == -INFINITY ? 0.f : expf(s[j][0] - mna);
    s[j][1] = s[j][1] == -INFINITY ? 0.f : expf(s[j][1] - mna);
    s[j][2] = s[j][2] == -INFINITY ? 0.f : expf(s[j][2] - mnb);
    s[j][3] = s[j][3] == -INFINITY ? 0.f : expf(s[j][3] - mnb);
    sa += s[j][0] + s[j][1];
    sb += s[j][2] + s[j][3];
  }
  sa += __shfl_xor_sync(0xffffffffu, sa, 1);
  sa += __shfl_xor_sync(0xffffffffu, sa, 2);
  sb += __shfl_xor_sync(0xffffffffu, sb, 1);
  sb += __shfl_xor_sync(0xffffffffu, sb, 2);
  la = la * ca + sa;
  lb = lb * cb + sb;
  ma = mna;
  mb = mnb;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    o[nt][0] *= ca; o[nt][1] *= ca; o[nt][2] *= cb; o[nt][3] *= cb;
  }
  // O += P V: P as A fragments (keys are the k dimension), V via ldmatrix.trans
#pragma unroll
  for (int kk = 0; kk < NJG / 2; ++kk) {
    uint32_t pf[4];
    pf[0] = pack_h2(s[2 * kk][0], s[2 * kk][1]);
    pf[1] = pack_h2(s[2 * kk][2], s[2 * kk][3]);
    pf[2] = pack_h2(s[2 * kk + 1][0], s[2 * kk + 1][1]);
    pf[3] = pack_h2(s[2 * kk + 1][2], s[2 * kk + 1][3]);
    const uint32_t vrow = smem_u32(sV + (koff + kk * 16 + (lane & 15)) * ROWB);
#pragma unroll
    for (int n0 = 0; n0 < NT; n0 += 4) {
      uint32_t vb[4][2];
#pragma unroll
      for (int u = 0; u < 4; ++u) ldsm_x2_trans(vb[u][0], vb[u][1], vrow + (n0 + u) * 16);
#pragma unroll
      for (int u = 0; u < 4; ++u) mma_f16_16816(o[n0 + u], pf, vb[u][0], vb[u][1]);
    }
  }
}

// One attention work unit of 4 warps (tid 0..127, warp = tid / 32): sequence
// b, kv head kvh, row block rb (rows row0 .. row0 + nrows - 1 of the pass,
// query vectors qv = r * GROUP + head), key split sp of ns over the 32-key
// chunks up to the block's last position.  Leaves the unnormalised output and
// the softmax (max, sum) of each query vector in smem as [64][kPartLd] floats
// (each warp its own query vectors; the caller synchronises before reading
// other warps'), and its row positions in s_pos[64].  bar() synchronises the
// 128 threads.
//
// Latency structure: a first round of loads brings the row positions, the
// sequence's first position in this pass and its page table row, none of
// which the producer of Q writes; the chunks wholly below that first
// position (keys and values of earlier passes) are requested next, and only
// then does the unit call wait_q() (the standalone kernel's wait on the
// previous kernel).  A second round brings Q, the remaining chunks follow, and
// NBUF - 1 chunks stay in flight while the warps compute on the oldest.
template <int HD, int GROUP, int NBUF, typename Bar, typename WaitQ>
__device__ AttnRows attn_unit(const AttnArgs& a, int b, int kvh, int rb, int sp, int ns, int M, uint8_t* smem,
                              int* s_pos, int tid, Bar bar, WaitQ wait_q) {
  static_assert(NBUF >= 2 && NBUF <= 4, "chunk ring of 2 to 4 buffers");
  using C = AttnCfg<HD, NBUF>;
  constexpr int RB = kMaxQV / GROUP;  // rows per block
  constexpr int NT = HD / 8;
  constexpr int NJ = kKeyChunk / 8;  // 8-key n-tiles per chunk
  const int warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, c4 = lane & 3;

  AttnRows R{0, 0, 0};
  int s0 = 0;
  if (b < a.batch) {
    s0 = a.rows_per_seq > 0 ? b * a.rows_per_seq : a.seq_row0[b];
    const int s1 = a.rows_per_seq > 0 ? s0 + a.rows_per_seq : a.seq_row0[b + 1];
    R.row0 = s0 + rb * RB;
    const int row_end = min(min(s1, R.row0 + RB), M);
    R.nrows = max(0, row_end - R.row0);
  }
  const int row0 = R.row0, nrows = R.nrows;
  const int nqv = nrows * GROUP;
  const int* pt = a.page_table + (size_t)(b < a.batch ? b : 0) * a.pt_ld;
  uint8_t* sQ = smem + C::kQOff;
  int* spg = reinterpret_cast<int*>(smem + C::kPageOff);
  const bool cached = a.pt_ld <= kAttnPageCache;

  // ---- first wave of loads: row positions, the sequence's first position, page table row ----
  const int pos_v = tid < nrows ? __ldcg(a.row_pos + row0 + tid) : -1;
  const int first_v = (tid == 0 && nrows > 0) ? __ldcg(a.row_pos + s0) : 0;
  int pg_v[kAttnPageCache / kAttnThreads];
#pragma unroll
  for (int k = 0; k < kAttnPageCache / kAttnThreads; ++k) {
    const int i = tid + k * kAttnThreads;
    pg_v[k] = (cached && i < a.pt_ld) ? __ldcg(pt + i) : -1;
  }
  if (tid < kMaxQV) s_pos[tid] = pos_v;
  if (tid == 0) spg[kAttnPageCache] = first_v;
#pragma unroll
  for (int k = 0; k < kAttnPageCache / kAttnThreads; ++k) spg[tid + k * kAttnThreads] = pg_v[k];
  bar();
  int maxpos = -1;
  for (int r = 0; r < nrows; ++r) maxpos = max(maxpos, s_pos[r]);
  const int first_new = spg[kAttnPageCache];  // keys from here on are written by this pass
  const int n_chunks = maxpos >= 0 ? maxpos / kKeyChunk + 1 : 0;
  R.n_chunks = n_chunks;
  // contiguous chunk ranges; the remainder goes to the first splits, so the
  // last one, which holds this pass's own keys (read only after wait_q),
  // has the fewest
  const int base = n_chunks / ns, rem = n_chunks % ns;
  const int c0 = sp * base + min(sp, rem), c1 = c0 + base + (sp < rem ? 1 : 0);
  const int n = c1 - c0;
  const int* pgs = cached ? spg : nullptr;

  // ---- chunks of earlier passes: in flight before Q is available ----
  auto kbuf = [&](int t) { return smem + (t % NBUF) * 2 * C::kTileBytes; };
  int issued = 0;
  for (; issued < n && issued < NBUF - 1 && (c0 + issued + 1) * kKeyChunk <= first_new; ++issued) {
    uint8_t* k = kbuf(issued);
    load_chunk<HD, NBUF>(a, pt, pgs, kvh, c0 + issued, maxpos, k, k + C::kTileBytes, tid);
    cp_async_commit();
  }
  wait_q();

  // ---- second wave of loads: Q ----
  // q is rewritten by every layer (by the previous kernel): L2 loads
  constexpr int kQIter = kMaxQV * (HD / 4) / kAttnThreads;  // 8 or 16 float4 per thread
  constexpr int kQGroup = kQIter < 8 ? kQIter : 8;
#pragma unroll 1
  for (int i0 = 0; i0 < kQIter; i0 += kQGroup) {
    float4 v[kQGroup];
#pragma unroll
    for (int u = 0; u < kQGroup; ++u) {
      const int i = tid + (i0 + u) * kAttnThreads;
      const int qv = i / (HD / 4), d4 = i % (HD / 4);
      v[u] = qv < nqv ? __ldcg(reinterpret_cast<const float4*>(a.q + (size_t)(row0 + qv / GROUP) * a.q_ld +
                                                               (kvh * GROUP + qv % GROUP) * HD) + d4)
                      : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kQGroup; ++u) {
      const int i = tid + (i0 + u) * kAttnThreads;
      const int qv = i / (HD / 4), d4 = i % (HD / 4);
      *reinterpret_cast<uint2*>(sQ + qv * C::kRowBytes + d4 * 8) =
          make_uint2(pack_h2(v[u].x, v[u].y), pack_h2(v[u].z, v[u].w));
    }
  }
  bar();
  // Warp roles.  Query vectors are tiled 16 to a warp.  In the two-buffer
  // form (passes with many units), when they fit in two warps and the unit
  // walks at least kKeyHalvesMinChunks chunks, the other two warps would
  // idle: instead warps 0-1 take keys 0-15 and warps 2-3 keys 16-31 of every
  // chunk, each pair with its own online-softmax state, and the pairs'
  // states are merged once after the last chunk.  (The four-buffer form of
  // batch-1 passes walks one or two chunks a unit and keeps one warp set.)
  constexpr bool kHalves = NBUF == 2;
  const int ng = (kHalves && (nqv + 15) / 16 <= 2 && n >= kKeyHalvesMinChunks) ? 2 : 1;
  const int qtile = ng == 2 ? (warp & 1) : warp;
  const int kgrp = ng == 2 ? (warp >> 1) : 0;
  const int qa = qtile * 16 + g, qb = qa + 8;
  const int posa = qa < nqv ? s_pos[qa / GROUP] : -1, posb = qb < nqv ? s_pos[qb / GROUP] : -1;

  // ---- K/V chunk ring: NBUF - 1 chunks in flight ----
  for (; issued < n && issued < NBUF - 1; ++issued) {
    uint8_t* k = kbuf(issued);
    load_chunk<HD, NBUF>(a, pt, pgs, kvh, c0 + issued, maxpos, k, k + C::kTileBytes, tid);
    cp_async_commit();
  }

  float o[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;
  float ma = -INFINITY, mb = -INFINITY, la = 0.f, lb = 0.f;
  const bool active = qtile * 16 < nqv;
  // ldmatrix.x4 row address of this lane in the warp's 16-row Q tile
  const uint32_t q_base = smem_u32(sQ) + (uint32_t)((qtile * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * C::kRowBytes +
                                                    ((lane >> 4) & 1) * 16);

  for (int t = 0; t < n; ++t) {
    const int ch = c0 + t;
    uint8_t* sK = kbuf(t);
    uint8_t* sV = sK + C::kTileBytes;
    cp_async_wait_upto(issued - 1 - t);  // chunk t has landed (this thread's copies)
    chunk_to_f16<HD, NBUF>(sK, sV, tid);
    bar();
    if (issued < n) {  // refill the buffer every warp finished with (chunk t - 1)
      uint8_t* k = kbuf(issued);
      load_chunk<HD, NBUF>(a, pt, pgs, kvh, c0 + issued, maxpos, k, k + C::kTileBytes, tid);
      cp_async_commit();
      ++issued;
    }
    if (active) {
      if constexpr (kHalves) {
        if (ng == 2)
          attn_chunk<HD, NJ / 2, C::kRowBytes>(sK, sV, kgrp * (kKeyChunk / 2), ch, q_base, posa, posb, a.scale, o,
                                               ma, mb, la, lb, lane);
        else
          attn_chunk<HD, NJ, C::kRowBytes>(sK, sV, 0, ch, q_base, posa, posb, a.scale, o, ma, mb, la, lb, lane);
      } else {
        attn_chunk<HD, NJ, C::kRowBytes>(sK, sV, 0, ch, q_base, posa, posb, a.scale, o, ma, mb, la, lb, lane);
      }
    }
  }
  bar();  // K/V and Q buffers are reused for the partial results below

  float* part = reinterpret_cast<float*>(smem);
  if (kHalves && ng == 2) {
    // Warps 2-3 hand their state to their twins in warps 0-1 (same lane, same
    // query vectors) through partial rows 32-63, which no push into this
    // CTA's receive area reaches: a unit walking kKeyHalvesMinChunks chunks
    // or more keeps the receive area above that many ring buffers.
    static_assert(2 * kKeyHalvesMinChunks * C::kTileBytes >= kMaxQV * C::kPartLd * 4,
                  "key-half merge rows overlap the push receive area");
    float* twin = part + (size_t)(kMaxQV / 2) * C::kPartLd;
    if (active && kgrp == 1) {
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int d = nt * 8 + 2 * c4;
        *reinterpret_cast<float2*>(twin + qa * C::kPartLd + d) = make_float2(o[nt][0], o[nt][1]);
        *reinterpret_cast<float2*>(twin + qb * C::kPartLd + d) = make_float2(o[nt][2], o[nt][3]);
      }
      if (c4 == 0) {
        *reinterpret_cast<float2*>(twin + qa * C::kPartLd + HD) = make_float2(ma, la);
        *reinterpret_cast<float2*>(twin + qb * C::kPartLd + HD) = make_float2(mb, lb);
      }
    }
    bar();
    if (active && kgrp == 0) {
      const float2 mla = *reinterpret_cast<const float2*>(twin + qa * C::kPartLd + HD);
      const float2 mlb = *reinterpret_cast<const float2*>(twin + qb * C::kPartLd + HD);
      const float na = fmaxf(ma, mla.x), nb = fmaxf(mb, mlb.x);
      const float sa0 = ma == -INFINITY ? 0.f : expf(ma - na), sa1 = mla.x == -INFINITY ? 0.f : expf(mla.x - na);
      const float sb0 = mb == -INFINITY ? 0.f : expf(mb - nb), sb1 = mlb.x == -INFINITY ? 0.f : expf(mlb.x - nb);
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int d = nt * 8 + 2 * c4;
        const float2 ta = *reinterpret_cast<const float2*>(twin + qa * C::kPartLd + d);
        const float2 tb = *reinterpret_cast<const float2*>(twin + qb * C::kPartLd + d);
        o[nt][0] = o[nt][0] * sa0 + ta.x * sa1;
        o[nt][1] = o[nt][1] * sa0 + ta.y * sa1;
        o[nt][2] = o[nt][2] * sb0 + tb.x * sb1;
        o[nt][3] = o[nt][3] * sb0 + tb.y * sb1;
      }
      la = la * sa0 + mla.y * sa1;
      lb = lb * sb0 + mlb.y * sb1;
      ma = na;
      mb = nb;
    }
  }

  // partial (unnormalised o, m, l) of this CTA in its own shared memory
  if (active && kgrp == 0) {
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int d = nt * 8 + 2 * c4;
      part[qa * C::kPartLd + d] = o[nt][0];
      part[qa * C::kPartLd + d + 1] = o[nt][1];
      part[qb * C::kPartLd + d] = o[nt][2];
      part[qb * C::kPartLd + d + 1] = o[nt][3];
    }
    if (c4 == 0) {
      part[qa * C::kPartLd + HD] = ma;
      part[qa * C::kPartLd + HD + 1] = la;
      part[qb * C::kPartLd + HD] = mb;
      part[qb * C::kPartLd + HD + 1] = lb;
    }
  }
  return R;
}

}  // namespace pard
