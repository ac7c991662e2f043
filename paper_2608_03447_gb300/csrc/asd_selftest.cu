// libasd: self-test of the failure detection (no counterpart in the paper).
//
// The pipeline kernels bound every mbarrier wait (about one second of
// %globaltimer) and record ASD_ERR_TIMEOUT in the workspace's error word when
// one gives up. asd_selftest_wait_timeout drives that path on purpose with a
// barrier that nothing signals, so a test can check it without faulting or
// hanging the GPU.
#include <cuda_runtime.h>
#include <stdint.h>

#include "asd.h"
#include "asd_device.cuh"

namespace {

using namespace asd_detail;

// One thread waits on an mbarrier that no one arrives at, through the bounded
// wait of the pipeline kernels; when it gives up, the error word records the
// timeout exactly as a stalled pipeline would.
__global__ void selftest_wait_kernel(unsigned int* error) {
  __shared__ unsigned long long bar;
  __shared__ int abort;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort = 0;
  }
  __syncthreads();
  if (threadIdx.x == 0 && !mbar_wait(&bar, 0, &abort)) atomicExch(error, static_cast<unsigned>(ASD_ERR_TIMEOUT));
}

}  // namespace

extern "C" {

int asd_selftest_wait_timeout(void* workspace, size_t workspace_bytes, asd_stream_t stream) {
  if (!workspace) return ASD_ERR_NULL;
  if (workspace_bytes < sizeof(unsigned int)) return ASD_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(workspace) % 16 != 0) return ASD_ERR_ALIGN;
  selftest_wait_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(static_cast<unsigned int*>(workspace));
  return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

}  // extern "C"
