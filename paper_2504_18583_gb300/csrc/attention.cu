// Multi-query-position GQA attention over the paged KV cache.
//
// Each new row (the K+1 verify rows, the a+K draft rows, or a prefill
// chunk) attends to every cached position up to its own position; the new
// rows' keys and values were written to the cache by the QKV epilogue, so
// the causal mask among them is just key_pos <= row_pos.
//
// Work unit: one sequence, one KV head, a block of rows times the query
// heads that share the KV head (<= 64 query vectors, 16 per warp), and one
// share of the key range.  The key range is split over the CTAs of one
// thread-block cluster (<= 8); each CTA walks its 64-key chunks with K/V
// pages double-buffered in shared memory (cp.async), computes S = Q K^T and
// O += P V on the tensor cores (mma.sync m16n8k16, bf16 inputs, fp32
// accumulators; Q and P carried as bf16 hi/lo pairs so the products keep
// fp32-level accuracy against the bf16 cache), and keeps the online-softmax
// state in registers.  The cluster then combines its partial (max, sum, O)
// through distributed shared memory, in rank order, and writes the output
// as bf16 hi/lo pairs in the packed activation layout of the O projection.
#include "common.cuh"
#include "internal.h"

namespace pard {

constexpr int kAttnThreads = 128;  // 4 warps x 16 query vectors
constexpr int kMaxQV = 64;
constexpr int kKeyChunk = 64;
constexpr int kMaxCluster = 8;

template <int HD>
struct AttnCfg {
  static constexpr int kRowBytes = HD * 2 + 16;             // padded smem row
  static constexpr int kTileBytes = kKeyChunk * kRowBytes;  // one K or V chunk
  static constexpr int kKV = 4 * kTileBytes;                // K and V, double-buffered
  static constexpr int kPart = kMaxQV * (HD + 2) * 4;       // partial (o, m, l) per CTA
  static constexpr int kSmem = (kKV > kPart ? kKV : kPart) + 256;
};

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x2_trans(uint32_t& r0, uint32_t& r1, uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];" : "=r"(r0), "=r"(r1) : "r"(addr));
}
// two fp32 -> bf16x2 (lower-index element in the low half), plus the bf16 remainders
__device__ __forceinline__ void split2(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat16 h0 = __float2bfloat16_rn(x0), h1 = __float2bfloat16_rn(x1);
  const __nv_bfloat16 l0 = __float2bfloat16_rn(x0 - __bfloat162float(h0));
  const __nv_bfloat16 l1 = __float2bfloat16_rn(x1 - __bfloat162float(h1));
  hi = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
  lo = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
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
__device__ __forceinline__ float ld_dsmem(const float* local, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(remote) : "memory");
  return v;
}

// K and V rows of one 64-key chunk into shared memory; positions past maxpos
// (masked anyway) and bad pages become zeros.
template <int HD>
__device__ __forceinline__ void load_chunk(const AttnArgs& a, const int* pt, int kvh, int chunk, int maxpos,
                                           uint8_t* sK, uint8_t* sV) {
  using C = AttnCfg<HD>;
  constexpr int kCh = HD * 2 / 16;
  for (int i = threadIdx.x; i < kKeyChunk * kCh; i += kAttnThreads) {
    const int key = i / kCh, ch = i % kCh;
    const int pos = chunk * kKeyChunk + key;
    uint8_t* dk = sK + key * C::kRowBytes + ch * 16;
    uint8_t* dv = sV + key * C::kRowBytes + ch * 16;
    int page = -1;
    if (pos <= maxpos) {
      if (pos / a.page_size < a.pt_ld) page = pt[pos / a.page_size];
      if (page < 0 || page >= a.n_pages) { set_status(a.status, ST_BAD_PAGE); page = -1; }
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
  cp_async_commit();
}

template <int HD, int GROUP>
__global__ void __launch_bounds__(kAttnThreads) attn_kernel(const __grid_constant__ AttnArgs a) {
  using C = AttnCfg<HD>;
  constexpr int RB = kMaxQV / GROUP;  // rows per block
  constexpr int KS = HD / 16;         // k-steps of QK^T
  constexpr int NT = HD / 8;          // n-tiles of O
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ int s_pos[kMaxQV];
  __shared__ float s_w[kMaxQV][kMaxCluster];

  pdl_wait();
  pdl_trigger();  // the next kernel may start streaming its weights now
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, c4 = lane & 3;
  const uint32_t rank = cluster_rank(), NS = cluster_size();
  const int group_idx = blockIdx.x / NS;
  const int rb = group_idx % a.row_blocks;
  const int kvh = (group_idx / a.row_blocks) % a.hkv;
  const int b = group_idx / (a.row_blocks * a.hkv);
  const int M = *a.m_dev;
  int row0 = 0, nrows = 0;
  if (b < a.batch) {
    row0 = a.seq_row0[b] + rb * RB;
    int row_end = min(a.seq_row0[b + 1], row0 + RB);
    row_end = min(row_end, M);
    nrows = max(0, row_end - row0);
  }
  const int nqv = nrows * GROUP;
  for (int r = threadIdx.x; r < kMaxQV; r += kAttnThreads) s_pos[r] = r < nrows ? a.row_pos[row0 + r] : -1;
  __syncthreads();
  int maxpos = -1;
  for (int r = 0; r < nrows; ++r) maxpos = max(maxpos, s_pos[r]);
  const int n_chunks = maxpos >= 0 ? maxpos / kKeyChunk + 1 : 0;
  const int c0 = (int)((long)rank * n_chunks / NS), c1 = (int)((long)(rank + 1) * n_chunks / NS);
  const int* pt = a.page_table + (size_t)(b < a.batch ? b : 0) * a.pt_ld;

  // Q fragments (rows 16*warp + g and + 8 of this CTA's query vectors), bf16 hi/lo
  const int qa = warp * 16 + g, qb = qa + 8;
  const int posa = qa < nqv ? s_pos[qa / GROUP] : -1, posb = qb < nqv ? s_pos[qb / GROUP] : -1;
  uint32_t qh[KS][4], ql[KS][4];
  {
    const float* qra = qa < nqv ? a.q + (size_t)(row0 + qa / GROUP) * a.q_ld + (kvh * GROUP + qa % GROUP) * HD : nullptr;
    const float* qrb = qb < nqv ? a.q + (size_t)(row0 + qb / GROUP) * a.q_ld + (kvh * GROUP + qb % GROUP) * HD : nullptr;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
      const int d0 = ks * 16 + 2 * c4;
      const float2 z = make_float2(0.f, 0.f);
      const float2 a0 = qra ? *reinterpret_cast<const float2*>(qra + d0) : z;
      const float2 a2 = qra ? *reinterpret_cast<const float2*>(qra + d0 + 8) : z;
      const float2 b0 = qrb ? *reinterpret_cast<const float2*>(qrb + d0) : z;
      const float2 b2 = qrb ? *reinterpret_cast<const float2*>(qrb + d0 + 8) : z;
      split2(a0.x, a0.y, qh[ks][0], ql[ks][0]);
      split2(b0.x, b0.y, qh[ks][1], ql[ks][1]);
      split2(a2.x, a2.y, qh[ks][2], ql[ks][2]);
      split2(b2.x, b2.y, qh[ks][3], ql[ks][3]);
    }
  }

  float o[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;
  float ma = -INFINITY, mb = -INFINITY, la = 0.f, lb = 0.f;
  const bool active = warp * 16 < nqv;

  if (c0 < c1) load_chunk<HD>(a, pt, kvh, c0, maxpos, smem, smem + C::kTileBytes);
  for (int ch = c0; ch < c1; ++ch) {
    const int buf = (ch - c0) & 1;
    const uint8_t* sK = smem + buf * 2 * C::kTileBytes;
    const uint8_t* sV = sK + C::kTileBytes;
    cp_async_wait_all();
    __syncthreads();
    if (ch + 1 < c1) {
      uint8_t* nK = smem + (buf ^ 1) * 2 * C::kTileBytes;
      load_chunk<HD>(a, pt, kvh, ch + 1, maxpos, nK, nK + C::kTileBytes);
    }
    if (active) {
      // S = Q K^T for 64 keys: 8 n-tiles of 8 keys
      float s[8][4];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
        const uint8_t* krow = sK + (j * 8 + g) * C::kRowBytes;
#pragma unroll
        for (int ks = 0; ks < KS; ++ks) {
          const uint32_t b0 = *reinterpret_cast<const uint32_t*>(krow + (ks * 16 + 2 * c4) * 2);
          const uint32_t b1 = *reinterpret_cast<const uint32_t*>(krow + (ks * 16 + 8 + 2 * c4) * 2);
          mma_bf16_16816(s[j], qh[ks], b0, b1);
          mma_bf16_16816(s[j], ql[ks], b0, b1);
        }
      }
      // scale, causal mask, online softmax (rows qa and qb)
      float mxa = -INFINITY, mxb = -INFINITY;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int kp = ch * kKeyChunk + j * 8 + 2 * c4;
        s[j][0] = kp <= posa ? s[j][0] * a.scale : -INFINITY;
        s[j][1] = kp + 1 <= posa ? s[j][1] * a.scale : -INFINITY;
        s[j][2] = kp <= posb ? s[j][2] * a.scale : -INFINITY;
        s[j][3] = kp + 1 <= posb ? s[j][3] * a.scale : -INFINITY;
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
      for (int j = 0; j < 8; ++j) {
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
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t ph[4], pl[4];
        split2(s[2 * kk][0], s[2 * kk][1], ph[0], pl[0]);
        split2(s[2 * kk][2], s[2 * kk][3], ph[1], pl[1]);
        split2(s[2 * kk + 1][0], s[2 * kk + 1][1], ph[2], pl[2]);
        split2(s[2 * kk + 1][2], s[2 * kk + 1][3], ph[3], pl[3]);
        const uint32_t vrow = smem_u32(sV + (kk * 16 + (lane & 15)) * C::kRowBytes);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          uint32_t b0, b1;
          ldsm_x2_trans(b0, b1, vrow + nt * 16);
          mma_bf16_16816(o[nt], ph, b0, b1);
          mma_bf16_16816(o[nt], pl, b0, b1);
        }
      }
    }
  }
  __syncthreads();  // K/V buffers are reused for the partial results below

  // partial (unnormalised o, m, l) of this CTA in its own shared memory
  float* part = reinterpret_cast<float*>(smem);
  if (active) {
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int d = nt * 8 + 2 * c4;
      part[qa * (HD + 2) + d] = o[nt][0];
      part[qa * (HD + 2) + d + 1] = o[nt][1];
      part[qb * (HD + 2) + d] = o[nt][2];
      part[qb * (HD + 2) + d + 1] = o[nt][3];
    }
    if (c4 == 0) {
      part[qa * (HD + 2) + HD] = ma;
      part[qa * (HD + 2) + HD + 1] = la;
      part[qb * (HD + 2) + HD] = mb;
      part[qb * (HD + 2) + HD + 1] = lb;
    }
  }
  cluster_sync();
  // combine in rank order; CTA `rank` finishes query vectors rank, rank+NS, ...
  for (int qv = (int)rank + (int)NS * (int)threadIdx.x; qv < nqv; qv += (int)NS * kAttnThreads) {
    float mx = -INFINITY;
    for (uint32_t r = 0; r < NS; ++r) mx = fmaxf(mx, ld_dsmem(part + qv * (HD + 2) + HD, r));
    float L = 0.f;
    for (uint32_t r = 0; r < NS; ++r) {
      const float mr = ld_dsmem(part + qv * (HD + 2) + HD, r);
      const float w = mr == -INFINITY ? 0.f : expf(mr - mx);
      s_w[qv][r] = w;
      L += ld_dsmem(part + qv * (HD + 2) + HD + 1, r) * w;
    }
    for (uint32_t r = 0; r < NS; ++r) s_w[qv][r] /= L;
  }
  __syncthreads();
  const int my_qv = nqv > (int)rank ? (nqv - (int)rank + (int)NS - 1) / (int)NS : 0;
  for (int i = threadIdx.x; i < my_qv * HD; i += kAttnThreads) {
    const int qv = (int)rank + (int)NS * (i / HD), d = i % HD;
    float acc = 0.f;
    for (uint32_t r = 0; r < NS; ++r) {
      const float w = s_w[qv][r];
      if (w != 0.f) acc += ld_dsmem(part + qv * (HD + 2) + d, r) * w;
    }
    const int m = row0 + qv / GROUP;
    const int col = (kvh * GROUP + qv % GROUP) * HD + d;
    __nv_bfloat16 hi, lo;
    split_bf16(acc, hi, lo);
    a.x_out[xpk(2 * m, col, a.x_rows)] = hi;
    a.x_out[xpk(2 * m + 1, col, a.x_rows)] = lo;
  }
  cluster_sync();  // peers may still be reading this CTA's partial
}

size_t attention_part_floats(int, int, int, int, int, int) { return 0; }

template <int HD, int GROUP>
static cudaError_t launch_attn_t(const AttnArgs& a, int grid, int cluster, cudaStream_t s, bool pdl) {
  static bool configured = false;
  const int smem = AttnCfg<HD>::kSmem;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(attn_kernel<HD, GROUP>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kAttnThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, attn_kernel<HD, GROUP>, a);
}

int attention_rows_per_block(int group) { return kMaxQV / group; }

// grid = groups * n_split CTAs; the n_split (<= 8) CTAs of one cluster share
// one (sequence, kv head, row block) and split its keys.
void launch_attention(const AttnArgs& a, int grid, cudaStream_t s, bool pdl) {
  const int group = a.hq / a.hkv;
  const int cl = a.n_split;
  cudaError_t e = cudaErrorInvalidValue;
  if (cl < 1 || cl > kMaxCluster || grid % cl) throw cudaErrorInvalidValue;
  if (a.hd == 128 && group == 4) e = launch_attn_t<128, 4>(a, grid, cl, s, pdl);
  else if (a.hd == 128 && group == 8) e = launch_attn_t<128, 8>(a, grid, cl, s, pdl);
  else if (a.hd == 64 && group == 4) e = launch_attn_t<64, 4>(a, grid, cl, s, pdl);
  else if (a.hd == 64 && group == 8) e = launch_attn_t<64, 8>(a, grid, cl, s, pdl);
  else if (a.hd == 128 && group == 2) e = launch_attn_t<128, 2>(a, grid, cl, s, pdl);
  else if (a.hd == 64 && group == 2) e = launch_attn_t<64, 2>(a, grid, cl, s, pdl);
  else if (a.hd == 128 && group == 1) e = launch_attn_t<128, 1>(a, grid, cl, s, pdl);
  else if (a.hd == 64 && group == 1) e = launch_attn_t<64, 1>(a, grid, cl, s, pdl);
  if (e != cudaSuccess) throw e;
}

}  // namespace pard
