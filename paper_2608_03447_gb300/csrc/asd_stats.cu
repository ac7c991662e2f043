// libasd: the verifier-side opportunity rate of Eq. 4 (Sec. 3.1), as counts.
//
// Over every draft-target mismatch position (x, i) of the given blocks, count
// those whose regret is at most tau and that are followed, inside the block,
// by p draft tokens equal to the target's argmax; also count |M|. One warp per
// block-request: lane j loads position j (one round of loads for the whole
// block), and ballots give the bit masks m (x_j == y*_j), d = ~m and
// R_t (r_j <= tau_t); S_p = AND_{k=1..p} (m >> k) (the next p tokens match;
// bits past the block are zero, which also enforces i + p <= K). Lanes then
// split the counters and count with popc. A CTA sums its warps in shared
// memory and adds to the caller's counters once per counter.
#include <cuda_runtime.h>
#include <stdint.h>

#include "asd.h"
#include "asd_device.cuh"
#include "asd_launch.cuh"

namespace {

using namespace asd_detail;

struct OpportunityArgs {
  float tau[ASD_OPPORTUNITY_MAX];
  int p[ASD_OPPORTUNITY_MAX];
  int ntau, np;
};

constexpr int kStatThreads = 256;
constexpr int kStatWarps = kStatThreads / 32;
constexpr unsigned kFullMask = 0xffffffffu;

__global__ void __launch_bounds__(kStatThreads)
    opportunity_kernel(const int32_t* __restrict__ row_argmax, const int32_t* __restrict__ draft,
                       const float* __restrict__ row_regret, const int32_t* __restrict__ status, int n, int K,
                       const __grid_constant__ OpportunityArgs a, unsigned long long* counts) {
  __shared__ unsigned int local[ASD_OPPORTUNITY_MAX * ASD_OPPORTUNITY_MAX + 1];
  __shared__ uint32_t s_mask[kStatWarps][2 * ASD_OPPORTUNITY_MAX];  // S_p per p, then R_t per tau
  const int ncount = a.ntau * a.np;
  for (int i = threadIdx.x; i <= ncount; i += blockDim.x) local[i] = 0u;
  // programmatic dependent launch: the next kernel may start its set-up now;
  // this one reads the verify outputs only once the kernel before it is done
  pdl_signal_dependents();
  pdl_wait_prerequisites();
  __syncthreads();

  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const long long b = static_cast<long long>(blockIdx.x) * kStatWarps + warp;
  if (b < n) {  // warp-uniform
    // every load of the block-request at once, the status included
    const bool mine = lane < K;
    int xj = 0, yj = 0;
    float rj = 0.0f;
    if (mine) {
      xj = draft[b * K + lane];
      yj = row_argmax[b * (K + 1) + lane];
      rj = row_regret[b * K + lane];
    }
    const int st = status ? status[b] : 0;
    if (st == 0) {
      const uint32_t m = __ballot_sync(kFullMask, mine && xj == yj);
      const uint32_t all = K >= 32 ? 0xffffffffu : ((1u << K) - 1u);
      const uint32_t d = ~m & all;  // M restricted to this block
      if (d) {
        for (int t = 0; t < a.ntau; ++t) {
          const uint32_t r = __ballot_sync(kFullMask, mine && rj <= a.tau[t]);
          if (lane == t) s_mask[warp][ASD_OPPORTUNITY_MAX + t] = r;
        }
        if (lane < a.np) {
          uint32_t sp = all;
          for (int k = 1; k <= a.p[lane] && sp; ++k) sp &= m >> k;
          s_mask[warp][lane] = sp;
        }
        __syncwarp();
        for (int c = lane; c < ncount; c += 32) {
          const int t = c / a.np, u = c - t * a.np;
          const int cnt = __popc(d & s_mask[warp][u] & s_mask[warp][ASD_OPPORTUNITY_MAX + t]);
          if (cnt) atomicAdd(&local[c], static_cast<unsigned>(cnt));
        }
        if (lane == 0) atomicAdd(&local[ncount], static_cast<unsigned>(__popc(d)));
      }
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i <= ncount; i += blockDim.x)
    if (local[i]) atomicAdd(&counts[i], static_cast<unsigned long long>(local[i]));
}

}  // namespace

extern "C" int asd_opportunity(const int32_t* row_argmax, const int32_t* draft, const float* row_regret,
                               const int32_t* status, int n, int K, const float* tau, int ntau,
                               const int32_t* p, int np, unsigned long long* counts, asd_stream_t stream) {
  if (n < 0 || K < 0 || K > ASD_MAX_K) return ASD_ERR_SHAPE;
  if (ntau < 1 || np < 1 || ntau > ASD_OPPORTUNITY_MAX || np > ASD_OPPORTUNITY_MAX) return ASD_ERR_SHAPE;
  if (!tau || !p || !counts) return ASD_ERR_NULL;
  OpportunityArgs a = {};
  a.ntau = ntau;
  a.np = np;
  for (int t = 0; t < ntau; ++t) {
    if (tau[t] != tau[t]) return ASD_ERR_CONTROL;
    a.tau[t] = tau[t];
  }
  for (int u = 0; u < np; ++u) {
    if (p[u] < 0) return ASD_ERR_CONTROL;
    a.p[u] = p[u];
  }
  if (n == 0 || K == 0) return ASD_OK;  // no position can mismatch
  if (!row_argmax || !draft || !row_regret) return ASD_ERR_NULL;
  const unsigned grid = static_cast<unsigned>((n + kStatWarps - 1) / kStatWarps);
  cudaLaunchAttribute attr;
  const cudaLaunchConfig_t cfg =
      pdl_config(dim3(grid), dim3(kStatThreads), reinterpret_cast<cudaStream_t>(stream), &attr);
  if (cudaLaunchKernelEx(&cfg, opportunity_kernel, row_argmax, draft, row_regret, status, n, K, a, counts) !=
      cudaSuccess)
    return ASD_ERR_CUDA;
  return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

// ---------------------------------------------------------------- cache and history advance (Sec. 3.3)
//
// After a block is verified, the caches and the token history advance along
// the emitted sequence only: committed[b][0..a]. One warp per request: lanes
// 0..a append the emitted tokens to the history, lane 0 advances the lengths.

namespace {

constexpr int kCommitThreads = 256;

__global__ void __launch_bounds__(kCommitThreads) commit_kernel(int B, int K, const int32_t* __restrict__ accepted_len,
                                                                const int32_t* __restrict__ committed, int pending,
                                                                int32_t* kv_len, int32_t* tokens, int32_t* token_len,
                                                                int max_tokens, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * (kCommitThreads / 32) + (threadIdx.x >> 5);
  if (b >= B) return;
  int a = accepted_len[b];
  a = a < 0 ? 0 : (a > K ? K : a);  // asd_verify writes 0..K; anything else is clamped (memory safety)
  const int len = tokens ? token_len[b] : 0;
  const bool room = !tokens || len + a + 1 <= max_tokens;
  if (tokens && room && lane <= a)
    tokens[static_cast<long long>(b) * max_tokens + len + lane] = committed[static_cast<long long>(b) * (K + 1) + lane];
  if (lane == 0) {
    if (status) status[b] = room ? 0 : ASD_STATUS_OVERFLOW;
    if (room) {
      if (tokens) token_len[b] = len + a + 1;
      if (kv_len) kv_len[b] += pending + a;
    }
  }
}

}  // namespace

extern "C" int asd_commit(int B, int K, const int32_t* accepted_len, const int32_t* committed, int pending,
                          int32_t* kv_len, int32_t* tokens, int32_t* token_len, int max_tokens, int32_t* status,
                          asd_stream_t stream) {
  if (B < 0 || K < 0 || K > ASD_MAX_K || (pending != 0 && pending != 1)) return ASD_ERR_SHAPE;
  if (B == 0) return ASD_OK;
  if (!accepted_len || !committed) return ASD_ERR_NULL;
  if (tokens && (!token_len || max_tokens < 1)) return ASD_ERR_NULL;
  // a plain launch: with programmatic dependent launch it measured slower
  // behind a kernel that does not trigger its dependents early
  constexpr int kWarps = kCommitThreads / 32;
  commit_kernel<<<static_cast<unsigned>((B + kWarps - 1) / kWarps), kCommitThreads, 0,
                  reinterpret_cast<cudaStream_t>(stream)>>>(B, K, accepted_len, committed, pending, kv_len, tokens,
                                                            token_len, max_tokens, status);
  return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}
