// libasd: combine step of the vocabulary-sharded verifier.
//
// Each vocabulary shard has reduced every target row to an asd_partial (key
// with the global index, exact top logit, the draft token's logit if the
// shard holds it). Here one warp per request merges row j's S partials in lane
// j -- the largest key wins (larger logit, then lower global index), its
// shard's top value comes with it, the draft logit comes from the shard that
// holds the draft token -- and runs the same selection as asd_verify, so the
// result equals the unsharded verify bit for bit.
#include <cuda_runtime.h>
#include <stdint.h>

#include "asd.h"
#include "asd_device.cuh"
#include "asd_launch.cuh"

namespace {

using namespace asd_detail;

constexpr int kCombineThreads = 256;

__global__ void __launch_bounds__(kCombineThreads) shard_combine_kernel(const asd_partial* __restrict__ parts,
                                                                        int S, const __grid_constant__ VerifyParams p) {
  const int lane = threadIdx.x & 31;
  const int warps = blockDim.x / 32;
  const int K = p.K, K1 = p.K + 1;
  const long long R = static_cast<long long>(p.B) * K1;
  pdl_signal_dependents();
  pdl_wait_prerequisites();  // the partials are read only once the kernel before this one is done
  for (int b = blockIdx.x * warps + (threadIdx.x >> 5); b < p.B; b += gridDim.x * warps) {
    BlockInputs in;
    in.key = 0ull;
    in.x = -1;
    in.zx = -INFINITY;
    in.top = 0.0f;
    in.top_exact = true;  // every shard sends its top value exactly as stored
    unsigned flags = 0u;
    if (lane < K1) {
      const long long row = static_cast<long long>(b) * K1 + lane;
      asd_partial best = parts[row];
      float zx = best.draft_logit;
      flags = best.flags;
      for (int s = 1; s < S; ++s) {
        const asd_partial q = parts[static_cast<long long>(s) * R + row];
        if (q.key > best.key) best = q;
        if (q.draft_logit != -INFINITY) zx = q.draft_logit;  // the shard that holds the draft token
        flags |= q.flags;
      }
      in.key = best.key;
      in.top = best.top;
      if (lane < K) {
        in.zx = zx;
        in.x = p.draft[static_cast<long long>(b) * K + lane];
      }
    }
    in.flags = __reduce_or_sync(kFull, flags);
    float budget = 0.0f, spent = 0.0f;
    if (lane == 0) {
      budget = p.ledger[b].budget;
      spent = p.ledger[b].spent;
    }
    budget = __shfl_sync(kFull, budget, 0);
    spent = __shfl_sync(kFull, spent, 0);
    bool wrote = false;
    select_block<float, false>(p, b, in, budget, spent, wrote, lane);
    if (lane == 0 && wrote) p.ledger[b].spent = spent;
  }
}

}  // namespace

extern "C" int asd_shard_combine(const asd_partial* partials, int S, int B, int K, int V, const int32_t* draft,
                                 asd_ledger* ledger, float gate, int cap, int32_t* accepted_len,
                                 int32_t* committed, int32_t* recovery, int32_t* row_argmax, float* row_regret,
                                 int32_t* status, asd_stream_t stream) {
  int rc = check_shape(B, K, V, ASD_F32);
  if (rc != ASD_OK) return rc;
  if (S < 1) return ASD_ERR_SHAPE;
  if (B == 0) return ASD_OK;
  if (!partials || !ledger || !accepted_len || !committed || !recovery) return ASD_ERR_NULL;
  if (K > 0 && !draft) return ASD_ERR_NULL;
  if (gate != gate || gate < 0.0f || cap < 0) return ASD_ERR_CONTROL;
  VerifyParams p = {};
  p.logits = nullptr;
  p.B = B;
  p.K = K;
  p.V = V;
  p.nblk = 1;
  p.v_total = V;
  p.draft = draft;
  p.ledger = ledger;
  p.gate = gate;
  p.cap = cap;
  p.accepted_len = accepted_len;
  p.committed = committed;
  p.recovery = recovery;
  p.row_argmax = row_argmax;
  p.row_regret = row_regret;
  p.status = status;
  constexpr int kWarps = kCombineThreads / 32;
  const unsigned grid = static_cast<unsigned>((B + kWarps - 1) / kWarps);
  cudaLaunchAttribute attr;
  const cudaLaunchConfig_t cfg =
      pdl_config(dim3(grid), dim3(kCombineThreads), reinterpret_cast<cudaStream_t>(stream), &attr);
  if (cudaLaunchKernelEx(&cfg, shard_combine_kernel, partials, S, p) != cudaSuccess) return ASD_ERR_CUDA;
  return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}
