// Host-side launch helpers shared by the step's kernel files: programmatic
// dependent launches and conditional graph bodies under stream capture.
#pragma once

#include <vector>

#include "ps_internal.cuh"

namespace ps {

// Launch with programmatic stream serialization: the kernel may be scheduled
// while its predecessor finishes (its CTAs wait in with_args until the
// predecessor's writes are visible), hiding the gap between dependent kernels.
template <typename... KArgs, typename... Args>
inline void launch_k(void (*kernel)(KArgs...), int grid, int block, size_t smem, cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3((unsigned)block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Under stream capture: append an 'if' conditional node to the graph being
// captured on st, and start capturing its body on aux.  Returns false (and
// the capture then fails as a whole) if any step is refused.
inline bool cond_open(cudaStream_t st, cudaStream_t aux, cudaGraphConditionalHandle h, cudaGraph_t* body_out = nullptr) {
  cudaStreamCaptureStatus cs;
  cudaGraph_t g = nullptr;
  const cudaGraphNode_t* deps = nullptr;
  size_t nd = 0;
  if (cudaStreamGetCaptureInfo(st, &cs, nullptr, &g, &deps, nullptr, &nd) != cudaSuccess ||
      cs != cudaStreamCaptureStatusActive)
    return false;
  std::vector<cudaGraphNode_t> dv(deps, deps + nd);
  cudaGraphNodeParams p{};
  p.type = cudaGraphNodeTypeConditional;
  p.conditional.handle = h;
  p.conditional.type = cudaGraphCondTypeIf;
  p.conditional.size = 1;
  cudaGraphNode_t node;
  const bool ok = cudaGraphAddNode(&node, g, dv.data(), nullptr, nd, &p) == cudaSuccess &&
                  cudaStreamUpdateCaptureDependencies(st, &node, nullptr, 1, cudaStreamSetCaptureDependencies) ==
                      cudaSuccess &&
                  cudaStreamBeginCaptureToGraph(aux, p.conditional.phGraph_out[0], nullptr, nullptr, 0,
                                                cudaStreamCaptureModeThreadLocal) == cudaSuccess;
  if (ok && body_out) *body_out = p.conditional.phGraph_out[0];
  return ok;
}
inline bool cond_close(cudaStream_t aux) {
  cudaGraph_t body = nullptr;
  return cudaStreamEndCapture(aux, &body) == cudaSuccess;
}
// A conditional handle of the graph being captured on st (default 0 at every
// launch of the graph).
inline bool cond_handle(cudaStream_t st, cudaGraphConditionalHandle* h) {
  cudaStreamCaptureStatus cs;
  cudaGraph_t g = nullptr;
  return cudaStreamGetCaptureInfo(st, &cs, nullptr, &g) == cudaSuccess && cs == cudaStreamCaptureStatusActive &&
         cudaGraphConditionalHandleCreate(h, g, 0, cudaGraphCondAssignDefault) == cudaSuccess;
}

}  // namespace ps
