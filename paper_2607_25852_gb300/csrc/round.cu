// round.cu -- a verification round per candidate budget as CUDA graphs, the
// budget chosen on the device (arxiv 2607.25852, Section 4.3: with a few
// budget ratios the reachable verification shapes form a small finite set, so
// a graph can be captured per (B, rho); and budget selection should leave the
// critical path instead of synchronising drafting and verification).
//
// The caller captures, per candidate budget T_m, everything that follows the
// allocation at that shape (its target forward over T_m packed rows, then
// spec_verify and spec_commit) into a graph instantiated for device launch.
// select_round_kernel, launched after spec_allocate inside a host-launched
// graph, reads the chosen T* where spec_allocate wrote it and tail-launches the
// matching graph: no host round trip between the budget choice and the rest of
// the round.
//
// spec_pack_rows gathers rows 0..n_i of each request from a full-depth buffer
// into the dense packed layout of an allocation: it stands in for a target
// forward whose output rows follow the packing.
//
// This translation unit is compiled as relocatable device code and linked with
// the device runtime (device-side cudaGraphLaunch).
#include <cuda_runtime.h>

#include "spec_internal.cuh"

namespace spec {

struct SelectParams {
  int M;
  int32_t T[SPEC_MAX_CANDIDATES];
  cudaGraphExec_t graph[SPEC_MAX_CANDIDATES];
  const int32_t* chosen_T;
  int32_t* launched;  // the candidate launched, -1 if none (or null)
  int32_t* status;
};

__global__ void select_round_kernel(const SelectParams p) {
  const int T = *p.chosen_T;
  int m = -1;
  for (int c = 0; c < p.M; ++c)
    if (p.T[c] == T) {
      m = c;
      break;
    }
  if (p.launched) *p.launched = m;
  if (m < 0) {
    report(p.status, SPEC_ERR_BAD_INPUT);  // T* is not a captured shape
    return;
  }
  if (cudaGraphLaunch(p.graph[m], cudaStreamGraphTailLaunch) != cudaSuccess) report(p.status, SPEC_ERR_CUDA);
}

// One CTA per packed destination row: find its request by binary search in
// row_offsets, copy the source row with 16-byte loads when aligned.
__global__ void __launch_bounds__(256) pack_rows_kernel(const char* src, size_t row_bytes, int B, int K,
                                                        const int32_t* row_offsets, char* dst, int R_dst,
                                                        int32_t* status) {
  const int r = blockIdx.x;
  pdl_wait_prerequisites();
  if (r >= R_dst) return;
  const int total = __ldg(row_offsets + B);
  if (r >= total) return;  // rows past the packed total are left as they are
  int lo = 0, hi = B;      // the request i with row_offsets[i] <= r < row_offsets[i + 1]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (__ldg(row_offsets + mid) <= r) lo = mid;
    else hi = mid;
  }
  const int j = r - __ldg(row_offsets + lo);
  if (j < 0 || j > K) {
    if (threadIdx.x == 0) report(status, SPEC_ERR_BAD_INPUT);
    return;
  }
  const char* s = src + ((size_t)lo * (K + 1) + j) * row_bytes;
  char* d = dst + (size_t)r * row_bytes;
  if (((reinterpret_cast<uintptr_t>(s) | reinterpret_cast<uintptr_t>(d) | row_bytes) & 15u) == 0) {
    const uint4* s4 = reinterpret_cast<const uint4*>(s);
    uint4* d4 = reinterpret_cast<uint4*>(d);
    for (size_t k = threadIdx.x; k < row_bytes / 16; k += blockDim.x) d4[k] = ldg_stream(s4 + k);
  } else {
    for (size_t k = threadIdx.x; k < row_bytes; k += blockDim.x) d[k] = s[k];
  }
}

}  // namespace spec

extern "C" int spec_graph_begin_capture(cudaStream_t stream) {
  if (!stream) return SPEC_ERR_INVALID_ARG;  // the legacy stream cannot be captured
  return cudaStreamBeginCapture(stream, cudaStreamCaptureModeRelaxed) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

extern "C" int spec_graph_end_capture(cudaStream_t stream, int device_launch, void** exec_out) {
  if (!exec_out) return SPEC_ERR_INVALID_ARG;
  *exec_out = nullptr;
  cudaGraph_t graph = nullptr;
  if (cudaStreamEndCapture(stream, &graph) != cudaSuccess || !graph) {
    cudaGetLastError();
    return SPEC_ERR_CUDA;
  }
  cudaGraphExec_t exec = nullptr;
  const unsigned long long flags = device_launch ? cudaGraphInstantiateFlagDeviceLaunch : 0ull;
  cudaError_t err = cudaGraphInstantiateWithFlags(&exec, graph, flags);
  cudaGraphDestroy(graph);
  if (err != cudaSuccess) {
    cudaGetLastError();
    return SPEC_ERR_CUDA;
  }
  if (device_launch && cudaGraphUpload(exec, stream) != cudaSuccess) {
    cudaGetLastError();
    cudaGraphExecDestroy(exec);
    return SPEC_ERR_CUDA;
  }
  *exec_out = exec;
  return SPEC_OK;
}

extern "C" int spec_graph_launch(void* exec, cudaStream_t stream) {
  if (!exec) return SPEC_ERR_INVALID_ARG;
  return cudaGraphLaunch(static_cast<cudaGraphExec_t>(exec), stream) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

extern "C" int spec_graph_destroy(void* exec) {
  if (!exec) return SPEC_OK;
  return cudaGraphExecDestroy(static_cast<cudaGraphExec_t>(exec)) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

extern "C" int spec_select_round(const int32_t* chosen_T, int M, const int32_t* cand_T, void* const* graphs,
                                 int32_t* launched_out, int32_t* status, cudaStream_t stream) {
  spec::NvtxRange range("spec_select_round");
  if (!chosen_T || M < 1 || M > SPEC_MAX_CANDIDATES || !cand_T || !graphs) return SPEC_ERR_INVALID_ARG;
  spec::SelectParams p{};
  p.M = M;
  for (int m = 0; m < M; ++m) {
    if (!graphs[m]) return SPEC_ERR_INVALID_ARG;
    p.T[m] = cand_T[m];
    p.graph[m] = static_cast<cudaGraphExec_t>(graphs[m]);
  }
  p.chosen_T = chosen_T;
  p.launched = launched_out;
  p.status = status;
  spec::select_round_kernel<<<1, 1, 0, stream>>>(p);
  return cudaGetLastError() == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

extern "C" int spec_pack_rows(const void* src, size_t row_bytes, int B, int K, const int32_t* row_offsets,
                              void* dst, int R_dst, int32_t* status, cudaStream_t stream) {
  spec::NvtxRange range("spec_pack_rows");
  if (!src || !dst || !row_offsets || row_bytes == 0 || B < 1 || K < 0 || K > SPEC_MAX_DRAFTS || R_dst < 1 ||
      (long long)B * (K + 1) > (1LL << 28))
    return SPEC_ERR_INVALID_ARG;
  const cudaError_t err =
      spec::launch_after_previous(spec::pack_rows_kernel, dim3((unsigned)R_dst), dim3(256), 0, stream,
                                  static_cast<const char*>(src), row_bytes, B, K, row_offsets,
                                  static_cast<char*>(dst), R_dst, status);
  if (err != cudaSuccess || cudaGetLastError() != cudaSuccess) return SPEC_ERR_CUDA;
  return SPEC_OK;
}
