// libasd: launch configuration shared by the small kernels that run after a
// verify call (the vocabulary-shard combine, the opportunity counts).
#pragma once

#include <cuda_runtime.h>

namespace asd_detail {

// A launch with programmatic dependent launch allowed: the kernel may become
// resident while the kernel before it on the stream finishes; it waits with
// griddepcontrol.wait before it reads anything that kernel wrote.
inline cudaLaunchConfig_t pdl_config(dim3 grid, dim3 block, cudaStream_t stream, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  attr->id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr->val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

}  // namespace asd_detail
