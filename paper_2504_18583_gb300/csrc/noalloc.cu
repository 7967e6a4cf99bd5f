// Acceptance from caller-given logits with no device allocation at all.
//
// Some callers cannot hand the library a workspace: runtimes without a device
// allocator, and engines that plan every byte of device memory ahead of time
// and forbid allocation (cudaMalloc or any allocating library call) on their
// serving path.  This entry point runs the same kernels as pard_set_logits +
// pard_accept_commit, but keeps all of their scratch -- the per-tile logit
// statistics, the per-sequence acceptance state and the resampling partials and
// counters -- in one file-scope device array of fixed size.  The caller passes
// only inputs and outputs.
#include <mutex>
#include <string>

#include "common.cuh"
#include "internal.h"

namespace pard {

void set_error(const std::string& msg);  // api.cu

namespace {

constexpr int kNaMaxBatch = 16;
constexpr int kNaMaxK = 8;
constexpr int kNaMaxVocab = 128256;
constexpr int kNaTiles = (kNaMaxVocab + kTileN - 1) / kTileN;
constexpr int kNaRowsT = kNaMaxBatch * (kNaMaxK + 1);  // target rows: B (K+1)
constexpr int kNaRowsD = kNaMaxBatch * kNaMaxK;        // draft rows: B K

constexpr size_t al(size_t x) { return (x + 255) & ~size_t(255); }
constexpr size_t kOffCall = 0;
constexpr size_t kOffStatsT = al(kOffCall + sizeof(CallArgs));
constexpr size_t kOffStatsIT = al(kOffStatsT + (size_t)kNaTiles * kNaRowsT * sizeof(float4));
constexpr size_t kOffStatsD = al(kOffStatsIT + (size_t)kNaTiles * kNaRowsT * sizeof(int2));
constexpr size_t kOffStatsID = al(kOffStatsD + (size_t)kNaTiles * kNaRowsD * sizeof(float4));
constexpr size_t kOffN = al(kOffStatsID + (size_t)kNaTiles * kNaRowsD * sizeof(int2));
constexpr size_t kOffPendCnt = al(kOffN + kNaMaxBatch * 4);
constexpr size_t kOffPend = al(kOffPendCnt + kNaMaxBatch * 4);
constexpr size_t kOffGen = al(kOffPend + kNaMaxBatch * (kNaMaxK + 1) * 4);
constexpr size_t kOffMaxNew = al(kOffGen + kNaMaxBatch * 4);
constexpr size_t kOffDone = al(kOffMaxNew + kNaMaxBatch * 4);
constexpr size_t kOffD = al(kOffDone + kNaMaxBatch * 4);
constexpr size_t kOffDnorm = al(kOffD + kNaMaxBatch * kNaMaxK * 4);
constexpr size_t kOffSampA = al(kOffDnorm + kNaMaxBatch * kNaMaxK * sizeof(float2));
constexpr size_t kOffSampNorm = al(kOffSampA + kNaMaxBatch * 4);
constexpr size_t kOffSampPart = al(kOffSampNorm + kNaMaxBatch * sizeof(float4));
constexpr size_t kOffSampCnt = al(kOffSampPart + (size_t)kNaMaxBatch * kResampleSplit * sizeof(float2));
constexpr size_t kNaBytes = al(kOffSampCnt + kNaMaxBatch * 4);  // about 6.3 MiB

}  // namespace

// The scratch itself: every GPU that loads the library holds these bytes
// until the process exits.  Host code must not use the symbol's host-side
// address; the device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNaBytes];

namespace {

std::mutex g_na_mu;
void* g_na_ptr[64] = {};

// Device address of the scratch on the current device, looked up once per
// device (with that device current) and cached.
void* na_scratch(std::string& err) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= 64) {
    err = std::string("pard_accept_noalloc: cudaGetDevice: ") + cudaGetErrorString(e);
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_na_mu);
  if (!g_na_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) {
      err = std::string("pard_accept_noalloc: cudaGetSymbolAddress: ") + cudaGetErrorString(e);
      return nullptr;
    }
    g_na_ptr[dev] = p;
  }
  return g_na_ptr[dev];
}

// Per-call state of the acceptance kernels: nothing generated yet, no length
// budget, resampling counters at zero.
__global__ void na_reset_state(DevState st, int B) {
  const int i = threadIdx.x;
  if (i < B) {
    st.n[i] = 1;
    st.pend_cnt[i] = 1;
    st.gen[i] = 0;
    st.max_new[i] = 1 << 30;
    st.done[i] = 0;
    st.samp_cnt[i] = 0;
  }
}

}  // namespace
}  // namespace pard

using namespace pard;

extern "C" pard_status pard_accept_noalloc(const float* d_target_logits, const float* d_draft_logits,
                                           const int32_t* d_draft, int32_t batch, int32_t K, int32_t vocab,
                                           int32_t sample, float temperature, uint64_t seed, uint64_t step,
                                           int32_t* d_accept_len, int32_t* d_emitted, void* stream) {
  if (!d_target_logits || !d_draft || !d_accept_len || !d_emitted || (sample && !d_draft_logits)) {
    set_error("pard_accept_noalloc: null argument");
    return PARD_ERR_ARG;
  }
  if (batch < 1 || batch > kNaMaxBatch || K < 1 || K > kNaMaxK || vocab < 8 || vocab > kNaMaxVocab ||
      vocab % 8) {
    set_error("pard_accept_noalloc: sizes exceed the static scratch (batch <= 16, 1 <= K <= 8, "
              "vocab <= 128256 and a multiple of 8)");
    return PARD_ERR_ARG;
  }
  if (!(temperature > 0.f)) {
    set_error("pard_accept_noalloc: temperature must be > 0");
    return PARD_ERR_ARG;
  }
  std::string err;
  uint8_t* base = reinterpret_cast<uint8_t*>(na_scratch(err));
  if (!base) {
    set_error(err);
    return PARD_ERR_CUDA;
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  CallArgs* call = reinterpret_cast<CallArgs*>(base + kOffCall);
  float4* stats_t = reinterpret_cast<float4*>(base + kOffStatsT);
  int2* stats_it = reinterpret_cast<int2*>(base + kOffStatsIT);
  float4* stats_d = reinterpret_cast<float4*>(base + kOffStatsD);
  int2* stats_id = reinterpret_cast<int2*>(base + kOffStatsID);
  DevState st;
  st.n = reinterpret_cast<int*>(base + kOffN);
  st.pend_cnt = reinterpret_cast<int*>(base + kOffPendCnt);
  st.pend = reinterpret_cast<int*>(base + kOffPend);
  st.gen = reinterpret_cast<int*>(base + kOffGen);
  st.max_new = reinterpret_cast<int*>(base + kOffMaxNew);
  st.done = reinterpret_cast<int*>(base + kOffDone);
  st.d = reinterpret_cast<int*>(base + kOffD);
  st.dnorm = reinterpret_cast<float2*>(base + kOffDnorm);
  st.samp_a = reinterpret_cast<int*>(base + kOffSampA);
  st.samp_norm = reinterpret_cast<float4*>(base + kOffSampNorm);
  st.samp_part = reinterpret_cast<float2*>(base + kOffSampPart);
  st.samp_cnt = reinterpret_cast<int*>(base + kOffSampCnt);
  st.kmax = K;
  const int tiles = (vocab + kTileN - 1) / kTileN;
  try {
    na_reset_state<<<1, kNaMaxBatch, 0, s>>>(st, batch);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) throw e;
    e = cudaMemcpyAsync(st.d, d_draft, (size_t)batch * K * 4, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) throw e;
    launch_set_call(call, CallArgs{seed, step, temperature, sample ? 1 : 0, K, 0}, s, false);
    launch_row_stats(d_target_logits, batch * (K + 1), vocab, tiles, kNaRowsT, call, -1, 1, stats_t, stats_it, s);
    AcceptArgs a;
    memset(&a, 0, sizeof(a));
    a.batch = batch; a.K = K; a.w_tiles = tiles; a.m_cap = kNaRowsT; a.vocab = vocab;
    a.stats = stats_t; a.stats_i = stats_it; a.logits = d_target_logits; a.dlogits = d_draft_logits;
    a.call = call; a.st = st;
    a.page_table = nullptr; a.pt_ld = 0; a.page_size = 16;
    a.accept_len = d_accept_len; a.emitted = d_emitted; a.kv_slots = nullptr; a.n_emit = nullptr;
    if (sample) {
      launch_row_stats(d_draft_logits, batch * K, vocab, tiles, kNaRowsD, call, -1, 1, stats_d, stats_id, s);
      SelectArgs sa;
      memset(&sa, 0, sizeof(sa));
      sa.mode = SEL_NORM_ONLY;
      sa.batch = batch; sa.K = K; sa.w_tiles = tiles; sa.m_cap = kNaRowsD; sa.vocab = vocab;
      sa.stats = stats_d; sa.stats_i = stats_id; sa.call = call; sa.st = st;
      launch_select(sa, s, false);
      launch_accept_sample(a, s, false);
    } else {
      launch_accept_greedy(a, s, false);
    }
  } catch (cudaError_t e) {
    set_error(std::string("pard_accept_noalloc: ") + cudaGetErrorString(e));
    return PARD_ERR_CUDA;
  }
  return PARD_OK;
}
