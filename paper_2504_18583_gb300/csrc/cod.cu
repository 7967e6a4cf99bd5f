// Conditional drop-token (COD) data construction (Section 3.2 and the
// appendix algorithm): which rows of the mask-token subtasks 2..K of one
// training sample are kept.
//
// Subtask k keeps n_k = round(N max(r^(k-1), r_min)) rows, chosen at random
// among its candidates: row j (position j, fed m_{k-2}, labelled x_{j+1}) is a
// candidate when its attention chain is complete -- subtask 2 rows always,
// subtask k >= 3 rows when row j-1 of subtask k-1 is kept (the integrity of
// prefix key-value states); rows j < k-2 have no chain.  The random choice
// keeps the candidates with the n_k smallest Philox words (stream 3, step =
// sample id, row k, v = j), ties to the lower j, so it is reproducible.
//
// One CTA per sample; subtasks run in order (each depends on the previous
// one's flags, kept in shared memory); within a subtask every candidate finds
// its rank among the candidates by a count over the subtask (n <= 4096).
#include "common.cuh"
#include "internal.h"

namespace pard {

constexpr int kCodThreads = 1024;
constexpr uint32_t kStreamCod = 3;

__global__ void __launch_bounds__(kCodThreads) cod_kernel(int N, int K, double r, double r_min, uint64_t seed,
                                                          uint64_t sample_id, int32_t* keep, int32_t* counts) {
  __shared__ uint32_t s_key[kCodMaxN];
  __shared__ uint8_t s_valid[kCodMaxN];
  __shared__ uint8_t s_keep[2][kCodMaxN];  // this subtask's and the previous one's flags
  __shared__ int s_cnt;
  const int tid = threadIdx.x;
  if (tid == 0) counts[0] = N;
  double g = 1.0;
  for (int k = 2; k <= K; ++k) {
    g *= r;
    const double gam = g > r_min ? g : r_min;
    const int n = (int)floor((double)N * gam + 0.5);
    const uint8_t* prev = s_keep[k & 1];
    uint8_t* cur = s_keep[(k & 1) ^ 1];
    if (tid == 0) s_cnt = 0;
    for (int j = tid; j < N; j += kCodThreads) {
      const bool v = j >= k - 2 && (k == 2 || prev[j - 1] != 0);
      s_valid[j] = v ? 1 : 0;
      s_key[j] = v ? philox_word(seed, kStreamCod, sample_id, 0u, (uint32_t)k, (uint32_t)j) : 0u;
    }
    __syncthreads();
    int mine = 0;
    for (int j = tid; j < N; j += kCodThreads) {
      int kept = 0;
      if (s_valid[j]) {
        const uint32_t kj = s_key[j];
        int rank = 0;
        for (int i = 0; i < N; ++i)
          rank += (s_valid[i] && (s_key[i] < kj || (s_key[i] == kj && i < j))) ? 1 : 0;
        kept = rank < n ? 1 : 0;
      }
      cur[j] = (uint8_t)kept;
      keep[(size_t)(k - 2) * N + j] = kept;
      mine += kept;
    }
    atomicAdd(&s_cnt, mine);
    __syncthreads();  // flags, count and the reads of s_valid / s_key are done
    if (tid == 0) counts[k - 1] = s_cnt;
    __syncthreads();  // s_cnt is reset by the next subtask
  }
}

void launch_cod(int N, int K, double r, double r_min, uint64_t seed, uint64_t sample_id, int32_t* keep,
                int32_t* counts, cudaStream_t s) {
  cod_kernel<<<1, kCodThreads, 0, s>>>(N, K, r, r_min, seed, sample_id, keep, counts);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) throw e;
}

}  // namespace pard
