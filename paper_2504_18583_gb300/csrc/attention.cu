// Multi-query-position GQA attention over the paged KV cache.
//
// Each new row (the K+1 verify rows, the a+K draft rows, or a prefill
// chunk) attends to every cached position up to its own position; the new
// rows' keys and values were written to the cache by the QKV epilogue, so
// the causal mask among them is just key_pos <= row_pos.
//
// Work unit (one CTA, 8 warps): one sequence, one KV head, a block of rows
// times the query heads that share the KV head (<= 64 query vectors), and a
// contiguous range of 64-key tiles.  K/V tiles are copied page by page into
// shared memory with cp.async (double-buffered); scores, the online softmax
// and P*V run on CUDA cores in fp32 (the step is bound by KV bytes and
// latency, not FLOPs, at these row counts).  When the key range is split,
// each split writes (max, sum, unnormalised output) and the last split to
// finish combines them in split order.  The output is written as bf16
// hi/lo pairs, the input format of the O projection.
#include "common.cuh"
#include "internal.h"

namespace pard {

constexpr int kAttnThreads = 256;
constexpr int kKeyTile = 64;
constexpr int kMaxQV = 64;

template <int HD>
struct AttnCfg {
  static constexpr int kRowBytes = HD * 2 + 16;  // padded smem row (bank-conflict free 16-byte reads)
  static constexpr int kTileBytes = kKeyTile * kRowBytes;
  static constexpr int kSmem = kMaxQV * HD * 4 + 4 * kTileBytes + 64;
};

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

template <int HD>
__device__ __forceinline__ void load_kv_tile(const AttnArgs& a, int b, int kvh, int kt, int maxpos, uint8_t* sK,
                                             uint8_t* sV) {
  using C = AttnCfg<HD>;
  constexpr int kChunksPerRow = HD * 2 / 16;
  for (int i = threadIdx.x; i < kKeyTile * kChunksPerRow; i += kAttnThreads) {
    const int key = i / kChunksPerRow, ch = i % kChunksPerRow;
    const int pos = kt * kKeyTile + key;
    uint8_t* dk = sK + key * C::kRowBytes + ch * 16;
    uint8_t* dv = sV + key * C::kRowBytes + ch * 16;
    int page = -1;
    if (pos <= maxpos) {
      if (pos / a.page_size < a.pt_ld) page = a.page_table[(size_t)b * a.pt_ld + pos / a.page_size];
      if (page < 0 || page >= a.n_pages) { set_status(a.status, ST_BAD_PAGE); page = -1; }
    }
    if (page < 0) {  // past the block's last position (masked) or a bad page: zeros, never NaN garbage
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
  constexpr int RB = kMaxQV / GROUP;          // rows per block
  constexpr int QPW = kMaxQV / 8;             // query vectors per warp
  constexpr int DPL = HD / 32;                // output dims per lane
  extern __shared__ __align__(16) uint8_t smem[];
  float* sq = reinterpret_cast<float*>(smem);                 // [kMaxQV][HD]
  uint8_t* sKV = smem + kMaxQV * HD * 4;                      // 2 x (K tile, V tile)
  int* sflag = reinterpret_cast<int*>(sKV + 4 * C::kTileBytes);

  pdl_wait();
  pdl_trigger();  // the next kernel may start streaming its weights now
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int idx = blockIdx.x;
  const int sp = idx % a.n_split; idx /= a.n_split;
  const int rb = idx % a.row_blocks; idx /= a.row_blocks;
  const int kvh = idx % a.hkv;
  const int b = idx / a.hkv;
  const int group_idx = blockIdx.x / a.n_split;
  if (b >= a.batch) return;
  const int M = *a.m_dev;
  const int row0 = a.seq_row0[b] + rb * RB;
  int row_end = a.seq_row0[b + 1];
  if (row_end > row0 + RB) row_end = row0 + RB;
  if (row_end > M) row_end = M;
  if (row0 >= row_end) return;
  const int nrows = row_end - row0;
  const int nqv = nrows * GROUP;

  int maxpos = 0;
  for (int r = 0; r < nrows; ++r) maxpos = max(maxpos, a.row_pos[row0 + r]);
  const int n_kt = maxpos / kKeyTile + 1;
  const int kt0 = (int)((long)sp * n_kt / a.n_split), kt1 = (int)((long)(sp + 1) * n_kt / a.n_split);

  // query vectors: qv = r * GROUP + g  ->  row row0 + r, head kvh * GROUP + g
  for (int i = threadIdx.x; i < nqv * HD; i += kAttnThreads) {
    const int qv = i / HD, d = i % HD;
    const int r = qv / GROUP, g = qv % GROUP;
    sq[qv * HD + d] = a.q[(size_t)(row0 + r) * a.q_ld + (kvh * GROUP + g) * HD + d];
  }

  float m_run[QPW], l_run[QPW], o[QPW][DPL];
  int qpos[QPW];
#pragma unroll
  for (int i = 0; i < QPW; ++i) {
    m_run[i] = -INFINITY;
    l_run[i] = 0.f;
    const int qv = warp + 8 * i;
    qpos[i] = qv < nqv ? a.row_pos[row0 + qv / GROUP] : -1;
#pragma unroll
    for (int d = 0; d < DPL; ++d) o[i][d] = 0.f;
  }

  if (kt0 < kt1) load_kv_tile<HD>(a, b, kvh, kt0, maxpos, sKV, sKV + C::kTileBytes);
  for (int kt = kt0; kt < kt1; ++kt) {
    const int buf = (kt - kt0) & 1;
    uint8_t* sK = sKV + buf * 2 * C::kTileBytes;
    uint8_t* sV = sK + C::kTileBytes;
    cp_async_wait_all();
    __syncthreads();
    if (kt + 1 < kt1) {
      uint8_t* nK = sKV + (buf ^ 1) * 2 * C::kTileBytes;
      load_kv_tile<HD>(a, b, kvh, kt + 1, maxpos, nK, nK + C::kTileBytes);
    }
    const int kp0 = kt * kKeyTile + lane, kp1 = kp0 + 32;
#pragma unroll
    for (int i = 0; i < QPW; ++i) {
      const int qv = warp + 8 * i;
      if (qv >= nqv) break;
      const float* qrow = sq + qv * HD;
      float s0 = 0.f, s1 = 0.f;
#pragma unroll 4
      for (int c8 = 0; c8 < HD / 8; ++c8) {
        const uint4 k0 = *reinterpret_cast<const uint4*>(sK + lane * C::kRowBytes + c8 * 16);
        const uint4 k1 = *reinterpret_cast<const uint4*>(sK + (lane + 32) * C::kRowBytes + c8 * 16);
        const float4 qa = *reinterpret_cast<const float4*>(qrow + c8 * 8);
        const float4 qb = *reinterpret_cast<const float4*>(qrow + c8 * 8 + 4);
        const float qf[8] = {qa.x, qa.y, qa.z, qa.w, qb.x, qb.y, qb.z, qb.w};
        const uint32_t kw0[4] = {k0.x, k0.y, k0.z, k0.w}, kw1[4] = {k1.x, k1.y, k1.z, k1.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          s0 += qf[2 * e] * __uint_as_float(kw0[e] << 16) + qf[2 * e + 1] * __uint_as_float(kw0[e] & 0xFFFF0000u);
          s1 += qf[2 * e] * __uint_as_float(kw1[e] << 16) + qf[2 * e + 1] * __uint_as_float(kw1[e] & 0xFFFF0000u);
        }
      }
      s0 = kp0 <= qpos[i] ? s0 * a.scale : -INFINITY;
      s1 = kp1 <= qpos[i] ? s1 * a.scale : -INFINITY;
      const float tmax = warp_max(fmaxf(s0, s1));
      const float m_new = fmaxf(m_run[i], tmax);
      if (m_new == -INFINITY) continue;
      const float corr = expf(m_run[i] - m_new);
      const float p0 = expf(s0 - m_new), p1 = expf(s1 - m_new);
      l_run[i] = l_run[i] * corr + warp_sum(p0 + p1);
      m_run[i] = m_new;
#pragma unroll
      for (int d = 0; d < DPL; ++d) o[i][d] *= corr;
#pragma unroll 8
      for (int j = 0; j < 32; ++j) {
        const float pj0 = __shfl_sync(0xffffffffu, p0, j);
        const float pj1 = __shfl_sync(0xffffffffu, p1, j);
        const uint8_t* v0 = sV + j * C::kRowBytes + lane * DPL * 2;
        const uint8_t* v1 = sV + (j + 32) * C::kRowBytes + lane * DPL * 2;
        if constexpr (DPL == 4) {
          const uint2 a0 = *reinterpret_cast<const uint2*>(v0), a1 = *reinterpret_cast<const uint2*>(v1);
          o[i][0] += pj0 * __uint_as_float(a0.x << 16) + pj1 * __uint_as_float(a1.x << 16);
          o[i][1] += pj0 * __uint_as_float(a0.x & 0xFFFF0000u) + pj1 * __uint_as_float(a1.x & 0xFFFF0000u);
          o[i][2] += pj0 * __uint_as_float(a0.y << 16) + pj1 * __uint_as_float(a1.y << 16);
          o[i][3] += pj0 * __uint_as_float(a0.y & 0xFFFF0000u) + pj1 * __uint_as_float(a1.y & 0xFFFF0000u);
        } else {
          const uint32_t a0 = *reinterpret_cast<const uint32_t*>(v0), a1 = *reinterpret_cast<const uint32_t*>(v1);
          o[i][0] += pj0 * __uint_as_float(a0 << 16) + pj1 * __uint_as_float(a1 << 16);
          o[i][1] += pj0 * __uint_as_float(a0 & 0xFFFF0000u) + pj1 * __uint_as_float(a1 & 0xFFFF0000u);
        }
      }
    }
    __syncthreads();
  }

  auto write_out = [&](int qv, const float* val) {
    const int r = qv / GROUP, g = qv % GROUP;
    const size_t col = (size_t)(kvh * GROUP + g) * HD + lane * DPL;
    const int m = row0 + r;
#pragma unroll
    for (int d = 0; d < DPL; ++d) {
      __nv_bfloat16 hi, lo;
      split_bf16(val[d], hi, lo);
      a.x_out[xpk(2 * m, (int)col + d, a.x_rows)] = hi;
      a.x_out[xpk(2 * m + 1, (int)col + d, a.x_rows)] = lo;
    }
  };

  if (a.n_split == 1) {
#pragma unroll
    for (int i = 0; i < QPW; ++i) {
      const int qv = warp + 8 * i;
      if (qv >= nqv) break;
      float val[DPL];
#pragma unroll
      for (int d = 0; d < DPL; ++d) val[d] = o[i][d] / l_run[i];
      write_out(qv, val);
    }
    return;
  }

  // split partials: [group][split][qv][HD + 2] = (o unnormalised, m, l)
  const size_t gbase = (size_t)group_idx * a.n_split * kMaxQV * (HD + 2);
#pragma unroll
  for (int i = 0; i < QPW; ++i) {
    const int qv = warp + 8 * i;
    if (qv >= nqv) break;
    float* p = a.part + gbase + ((size_t)sp * kMaxQV + qv) * (HD + 2);
#pragma unroll
    for (int d = 0; d < DPL; ++d) p[lane * DPL + d] = o[i][d];
    if (lane == 0) { p[HD] = m_run[i]; p[HD + 1] = l_run[i]; }
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int old = atomicAdd(&a.counters[group_idx], 1);
    *sflag = (old == a.n_split - 1);
  }
  __syncthreads();
  if (!*sflag) return;
  __threadfence();
  // combine the splits in split order: w_s = exp(m_s - M) / sum_s l_s exp(m_s - M)
  const int ns = a.n_split;
  float* sw = sq;                       // [nqv][ns] weights (q is no longer needed)
  float* sl = sq + kMaxQV * ns;         // [nqv][ns] split sums
  for (int i = threadIdx.x; i < nqv * ns; i += kAttnThreads) {
    const int qv = i / ns, s2 = i % ns;
    const float* p = a.part + gbase + ((size_t)s2 * kMaxQV + qv) * (HD + 2);
    sw[i] = __ldcg(p + HD);
    sl[i] = __ldcg(p + HD + 1);
  }
  __syncthreads();
  for (int qv = threadIdx.x; qv < nqv; qv += kAttnThreads) {
    float mx = -INFINITY;
    for (int s2 = 0; s2 < ns; ++s2) mx = fmaxf(mx, sw[qv * ns + s2]);
    float L = 0.f;
    for (int s2 = 0; s2 < ns; ++s2) {
      const float m2 = sw[qv * ns + s2];
      const float w = m2 == -INFINITY ? 0.f : expf(m2 - mx);
      sw[qv * ns + s2] = w;
      L += sl[qv * ns + s2] * w;
    }
    for (int s2 = 0; s2 < ns; ++s2) sw[qv * ns + s2] /= L;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < nqv * HD; i += kAttnThreads) {
    const int qv = i / HD, d = i % HD;
    float acc = 0.f;
#pragma unroll 4
    for (int s2 = 0; s2 < ns; ++s2) {
      const float w = sw[qv * ns + s2];
      if (w != 0.f) acc += __ldcg(a.part + gbase + ((size_t)s2 * kMaxQV + qv) * (HD + 2) + d) * w;
    }
    const int r = qv / GROUP, g = qv % GROUP;
    const int m = row0 + r;
    const size_t col = (size_t)(kvh * GROUP + g) * HD + d;
    __nv_bfloat16 hi, lo;
    split_bf16(acc, hi, lo);
    a.x_out[xpk(2 * m, (int)col, a.x_rows)] = hi;
    a.x_out[xpk(2 * m + 1, (int)col, a.x_rows)] = lo;
  }
  if (threadIdx.x == 0) a.counters[group_idx] = 0;
}

size_t attention_part_floats(int batch, int hkv, int row_blocks, int n_split, int /*qv*/, int hd) {
  return (size_t)batch * hkv * row_blocks * n_split * kMaxQV * (hd + 2);
}

template <int HD, int GROUP>
static cudaError_t launch_attn_t(const AttnArgs& a, int grid, cudaStream_t s, bool pdl) {
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
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, attn_kernel<HD, GROUP>, a);
}

int attention_rows_per_block(int group) { return kMaxQV / group; }

void launch_attention(const AttnArgs& a, int grid, cudaStream_t s, bool pdl) {
  const int group = a.hq / a.hkv;
  cudaError_t e = cudaErrorInvalidValue;
  if (a.hd == 128 && group == 4) e = launch_attn_t<128, 4>(a, grid, s, pdl);
  else if (a.hd == 128 && group == 8) e = launch_attn_t<128, 8>(a, grid, s, pdl);
  else if (a.hd == 64 && group == 4) e = launch_attn_t<64, 4>(a, grid, s, pdl);
  else if (a.hd == 64 && group == 8) e = launch_attn_t<64, 8>(a, grid, s, pdl);
  else if (a.hd == 128 && group == 2) e = launch_attn_t<128, 2>(a, grid, s, pdl);
  else if (a.hd == 64 && group == 2) e = launch_attn_t<64, 2>(a, grid, s, pdl);
  else if (a.hd == 128 && group == 1) e = launch_attn_t<128, 1>(a, grid, s, pdl);
  else if (a.hd == 64 && group == 1) e = launch_attn_t<64, 1>(a, grid, s, pdl);
  if (e != cudaSuccess) throw e;
}

}  // namespace pard
