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
// thread-block cluster (<= 16); each CTA walks its 32-key chunks with K/V
// pages double-buffered in shared memory (cp.async), computes S = Q K^T and
// O += P V on the tensor cores (mma.sync m16n8k16, fp16 inputs, fp32
// accumulators: Q and P rounded to fp16, the bf16 K/V converted to fp16 in
// shared memory, which is exact in fp16's range), and keeps the online-softmax
// state in registers.  The cluster then combines its partial (max, sum, O)
// through distributed shared memory, in rank order, and writes the output
// as bf16 hi/lo pairs in the packed activation layout of the O projection.
#include "attn_core.cuh"

namespace pard {

// K/V chunk ring: NBUF = 4 buffers (three chunks in flight, ~87 KB at
// hd = 128, two CTAs per SM) when a pass has few units, as at batch 1; NBUF =
// 2 (one chunk in flight, four CTAs per SM) when its units fill the SMs more
// than twice over (ragged batches with long contexts), where the latency of
// a unit's dependent steps is hidden by the other CTAs' warps instead.
template <int HD, int GROUP, int NBUF>
__global__ void __launch_bounds__(kAttnThreads) attn_kernel(const __grid_constant__ AttnArgs a) {
  using C = AttnCfg<HD, NBUF>;
  constexpr int LD = C::kPartLd;
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ int s_pos[kMaxQV];
  __shared__ __align__(8) uint64_t s_recv;  // push combine: this CTA's incoming partials
  __shared__ int s_flag;                    // never raised: the wait below has no other role to abort it

  const uint32_t rank = cluster_rank(), NS = cluster_size();
  if (threadIdx.x == 0) {
    mbar_init(&s_recv, 1);
    s_flag = 0;
    fence_barrier_init();
  }
  // first cluster barrier: every CTA's s_recv is initialised (waited on
  // before any partial is pushed)
  cluster_arrive_relaxed();
  const int group_idx = blockIdx.x / NS;
  const int rb = group_idx % a.row_blocks;
  const int kvh = (group_idx / a.row_blocks) % a.hkv;
  const int b = group_idx / (a.row_blocks * a.hkv);
  // Row plan, positions, page tables and the keys and values of earlier
  // passes are written before the previous kernel (the QKV projection), which
  // had itself waited for them before it let this grid start: the unit reads
  // them before waiting, and Q after.
  const int M = a.rows_per_seq > 0 ? a.batch * a.rows_per_seq : __ldcg(a.m_dev);
  const AttnRows R = attn_unit<HD, GROUP, NBUF>(a, b, kvh, rb, (int)rank, (int)NS, M, smem, s_pos,
                                                     threadIdx.x, [] { __syncthreads(); }, [] { pdl_wait(); });
  const int row0 = R.row0, nqv = R.nrows * GROUP;
  // the next kernel may start streaming its weights once the key/value reads
  // are done: earlier, its bulk loads would queue ahead of them
  pdl_trigger();
  float* part = reinterpret_cast<float*>(smem);

  // Push combine: CTA o finishes query vectors [o cnt, (o + 1) cnt).  Every
  // CTA copies those rows of its partial into CTA o's shared memory with one
  // bulk copy, counted on o's s_recv, so a CTA waits only for its own inputs
  // and reads them locally.  The receive area is the part of the K/V ring that
  // no CTA of the cluster uses (each walks at most max_n chunks) above this
  // CTA's own partial; when it does not fit, the cluster pulls instead.
  const int cnt = (nqv + (int)NS - 1) / (int)NS;
  const int max_n = (R.n_chunks + (int)NS - 1) / (int)NS;
  // the partial rows written: every active warp writes all 16 of its rows
  const uint32_t part_bytes = (uint32_t)((nqv + 15) / 16 * 16) * LD * 4;
  const uint32_t ring_used = (uint32_t)max_n * 2 * C::kTileBytes;
  const uint32_t recv_off = ((ring_used > part_bytes ? ring_used : part_bytes) + 127) & ~127u;
  const uint32_t recv_bytes = NS * (uint32_t)cnt * LD * 4;
  const bool push = NS > 1 && recv_off + recv_bytes <= (uint32_t)C::kKV;
  if (a.paths && rank == 0 && threadIdx.x == 0)
    atomicOr(a.paths, (NS == 1 ? 0u : push ? kAttnPathPush : kAttnPathPull) | (NBUF == 2 ? kAttnPathRing2 : 0u) |
                          (1u << (kAttnPathSplit0 + NS)));
  // every thread's partial writes, ordered before the async-proxy reads of
  // the bulk copies below, and every warp's partial in shared memory
  fence_proxy_async_smem();
  __syncthreads();
  cluster_wait();  // first barrier
  if (push) {
    float* recv = reinterpret_cast<float*>(smem + recv_off);  // [NS][cnt][LD]
    const int my0 = (int)rank * cnt;
    const int my_n = max(0, min(nqv, my0 + cnt) - my0);
    if (threadIdx.x == 0 && my_n > 0) mbar_arrive_expect_tx(&s_recv, NS * (uint32_t)my_n * LD * 4);
    if (threadIdx.x < NS) {
      const uint32_t o = threadIdx.x;
      const int r0 = (int)o * cnt, rn = max(0, min(nqv, r0 + cnt) - r0);
      if (rn > 0) {
        bulk_copy_to_peer(mapa_shared(recv + (size_t)rank * cnt * LD, o), part + (size_t)r0 * LD,
                          (uint32_t)rn * LD * 4, mapa_shared(&s_recv, o));
        bulk_commit();
        bulk_wait_read_all();
      }
    }
    // second barrier, arrive: this CTA's pushes are issued and their sources read
    cluster_arrive();
    bool ok = my_n == 0 || mbar_wait(&s_recv, 0, &s_flag);
    if (!ok && threadIdx.x == 0) set_status(a.status, ST_TIMEOUT_EPI);
    // every copy out of this CTA's partial has been read (its issuers waited
    // before the barrier below), so the partial's area is free for the weights
    ok = __syncthreads_and(ok);
    if (ok) {
      // split weights exp(m_s - max) / L of each finished row: a half-warp per
      // row, lane s holding split s, max and sum by shuffles
      float* sw = part;  // [my_n][kMaxCluster]
      const int sr = threadIdx.x & 15;
      for (int r0 = 0; r0 < my_n; r0 += kAttnThreads / 16) {
        const int r = r0 + (int)(threadIdx.x >> 4);
        const bool live = r < my_n && sr < (int)NS;
        const float m = live ? recv[((size_t)sr * cnt + r) * LD + HD] : -INFINITY;
        float mx = m;
#pragma unroll
        for (int off = 8; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off, 16));
        const float w = m == -INFINITY ? 0.f : expf(m - mx);
        float L = live ? recv[((size_t)sr * cnt + r) * LD + HD + 1] * w : 0.f;
#pragma unroll
        for (int off = 8; off > 0; off >>= 1) L += __shfl_xor_sync(0xffffffffu, L, off, 16);
        if (live) sw[r * kMaxCluster + sr] = w / L;
      }
      __syncthreads();
      for (int i = threadIdx.x; i < my_n * (HD / 4); i += kAttnThreads) {
        const int r = i / (HD / 4), d4 = i % (HD / 4);
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
        for (int s2 = 0; s2 < (int)NS; ++s2) {
          const float w = sw[r * kMaxCluster + s2];
          const float4 v = *reinterpret_cast<const float4*>(recv + ((size_t)s2 * cnt + r) * LD + 4 * d4);
          acc.x += v.x * w;
          acc.y += v.y * w;
          acc.z += v.z * w;
          acc.w += v.w * w;
        }
        const int qv = my0 + r;
        store_pair4(a.x_out, row0 + qv / GROUP, (kvh * GROUP + qv % GROUP) * HD + 4 * d4, a.x_rows, acc);
      }
    }
    // second barrier, wait: no peer copies into this CTA any more
    cluster_wait();
    return;
  }
  cluster_sync();
  // Pull combine, in rank order; CTA `rank` finishes query vectors rank,
  // rank+NS, ...  Each thread takes one output pair (qv, d..d+1) at a time
  // and requests every rank's (max, sum) and partial values before using any,
  // so a round of work is one distributed-shared-memory round trip.
  const int my_qv = nqv > (int)rank ? (nqv - (int)rank + (int)NS - 1) / (int)NS : 0;
  const int n_items = my_qv * (HD / 2);
  for (int i = threadIdx.x; i < n_items; i += kAttnThreads) {
    const int qv = (int)rank + (int)NS * (i / (HD / 2)), d = 2 * (i % (HD / 2));
    float2 ml[kMaxCluster], pv[kMaxCluster];
#pragma unroll
    for (int r = 0; r < kMaxCluster; ++r) {
      const bool live = r < (int)NS;
      ml[r] = live ? ld_dsmem2(part + qv * LD + HD, (uint32_t)r) : make_float2(-INFINITY, 0.f);
      pv[r] = live ? ld_dsmem2(part + qv * LD + d, (uint32_t)r) : make_float2(0.f, 0.f);
    }
    float mx = -INFINITY;
#pragma unroll
    for (int r = 0; r < kMaxCluster; ++r) mx = fmaxf(mx, ml[r].x);
    float L = 0.f;
    float2 acc = make_float2(0.f, 0.f);
#pragma unroll
    for (int r = 0; r < kMaxCluster; ++r) {
      const float w = ml[r].x == -INFINITY ? 0.f : expf(ml[r].x - mx);
      L += ml[r].y * w;
      acc.x += pv[r].x * w;
      acc.y += pv[r].y * w;
    }
    const int m = row0 + qv / GROUP;
    const int col = (kvh * GROUP + qv % GROUP) * HD + d;
    __nv_bfloat16 h0, l0, h1, l1;
    split_bf16(acc.x / L, h0, l0);
    split_bf16(acc.y / L, h1, l1);
    *reinterpret_cast<uint32_t*>(a.x_out + xpk(2 * m, col, a.x_rows)) =
        (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
    *reinterpret_cast<uint32_t*>(a.x_out + xpk(2 * m + 1, col, a.x_rows)) =
        (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
  }
  cluster_sync();  // peers may still be reading this CTA's partial
}

template <int HD, int GROUP, int NBUF>
static cudaError_t launch_attn_nb(const AttnArgs& a, int grid, int cluster, cudaStream_t s, bool pdl) {
  static bool configured = false;
  const int smem = AttnCfg<HD, NBUF>::kSmem;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(attn_kernel<HD, GROUP, NBUF>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(attn_kernel<HD, GROUP, NBUF>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
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
  return cudaLaunchKernelEx(&cfg, attn_kernel<HD, GROUP, NBUF>, a);
}

template <int HD, int GROUP>
static cudaError_t launch_attn_t(const AttnArgs& a, int grid, int cluster, cudaStream_t s, bool pdl) {
  return a.nbuf == 2 ? launch_attn_nb<HD, GROUP, 2>(a, grid, cluster, s, pdl)
                     : launch_attn_nb<HD, GROUP, 4>(a, grid, cluster, s, pdl);
}

int attention_rows_per_block(int group) { return kMaxQV / group; }

// grid = groups * n_split CTAs; the n_split (<= 16) CTAs of one cluster share
// one (sequence, kv head, row block) and split its keys.  A cluster above 8
// CTAs that the GPU cannot place falls back to 8.
static cudaError_t launch_attn_any(const AttnArgs& a, int group, int grid, int cl, cudaStream_t s, bool pdl);

void launch_attention(const AttnArgs& a, int grid, cudaStream_t s, bool pdl) {
  const int group = a.hq / a.hkv;
  const int cl = a.n_split;
  if (cl < 1 || cl > kMaxCluster || grid % cl) throw cudaErrorInvalidValue;
  cudaError_t e = launch_attn_any(a, group, grid, cl, s, pdl);
  if (e != cudaSuccess && cl > 8) {
    (void)cudaGetLastError();
    e = launch_attn_any(a, group, grid / cl * 8, 8, s, pdl);
  }
  if (e != cudaSuccess) throw e;
}

static cudaError_t launch_attn_any(const AttnArgs& a, int group, int grid, int cl, cudaStream_t s, bool pdl) {
  cudaError_t e = cudaErrorInvalidValue;
  if (a.hd == 128 && group == 4) e = launch_attn_t<128, 4>(a, grid, cl, s, pdl);
  else if (a.hd == 128 && group == 8) e = launch_attn_t<128, 8>(a, grid, cl, s, pdl);
  else if (a.hd == 64 && group == 4) e = launch_attn_t<64, 4>(a, grid, cl, s, pdl);
  else if (a.hd == 64 && group == 8) e = launch_attn_t<64, 8>(a, grid, cl, s, pdl);
  else if (a.hd == 128 && group == 2) e = launch_attn_t<128, 2>(a, grid, cl, s, pdl);
  else if (a.hd == 64 && group == 2) e = launch_attn_t<64, 2>(a, grid, cl, s, pdl);
  else if (a.hd == 128 && group == 1) e = launch_attn_t<128, 1>(a, grid, cl, s, pdl);
  else if (a.hd == 64 && group == 1) e = launch_attn_t<64, 1>(a, grid, cl, s, pdl);
  return e;
}

}  // namespace pard
