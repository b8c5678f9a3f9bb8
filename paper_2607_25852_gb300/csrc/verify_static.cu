// verify_static.cu -- spec_verify for callers that cannot allocate device
// memory.
//
// Some callers of this library are not free to allocate GPU memory.  An
// inference engine that owns every byte of device memory through its own pool
// may forbid allocations made behind its back: under a tight memory budget
// such an allocation can fail, and either way it escapes the engine's memory
// accounting.  Code on a latency-critical path may not be allowed to call
// cudaMalloc at all, because cudaMalloc can synchronise the device.  These
// callers still pass their own inputs and outputs, but they cannot supply the
// scratch workspace that spec_verify needs.
//
// spec_verify_static gives them that scratch from a fixed array in device
// memory that belongs to this library: SPEC_STATIC_SCRATCH_BYTES bytes,
// reserved on every GPU that loads the library and held until the process
// exits.  Nothing here allocates.
#include <mutex>

#include "spec_internal.cuh"

namespace {

// The scratch itself.  Zero at module load; each call clears the part that
// must start at zero.
static __device__ __align__(256) unsigned char g_verify_scratch[SPEC_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 256;
std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_verify_scratch on the current device.  In host code the
// name g_verify_scratch only denotes a host-side stand-in, so the address is
// looked up once per device, with that device current, and cached.
int scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SPEC_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_scratch_ptr[dev] == nullptr) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_verify_scratch) != cudaSuccess || ptr == nullptr)
      return SPEC_ERR_CUDA;
    g_scratch_ptr[dev] = ptr;
  }
  *out = g_scratch_ptr[dev];
  return SPEC_OK;
}

}  // namespace

extern "C" int spec_verify_static(const void* logits, int logits_dtype, const int32_t* row_offsets,
                                  const int32_t* depth, const int32_t* draft_tokens, const void* q,
                                  int q_dtype, int B, int K, int V, float temperature,
                                  const uint64_t* seeds, const uint64_t* request_ids,
                                  const int64_t* pos_base, int32_t* accepted_len_out,
                                  int32_t* out_tokens, float* p_draft_out, float* row_stats_out,
                                  int32_t* status, cudaStream_t stream) {
  const size_t need = spec_verify_workspace(B, K, V);
  if (need == 0) return SPEC_ERR_INVALID_ARG;
  if (need > (size_t)SPEC_STATIC_SCRATCH_BYTES) return SPEC_ERR_TOO_LARGE;
  void* scratch = nullptr;
  const int rc = scratch_address(&scratch);
  if (rc != SPEC_OK) return rc;
  // The arrival counters must be zero when a call starts; clear them rather
  // than rely on what the previous call left behind.
  const spec::VerifyGeometry g = spec::verify_geometry(B, K, V);
  if (cudaMemsetAsync(static_cast<char*>(scratch) + g.counters_off, 0, need - g.counters_off,
                      stream) != cudaSuccess)
    return SPEC_ERR_CUDA;
  return spec_verify(logits, logits_dtype, row_offsets, depth, draft_tokens, q, q_dtype, B, K, V,
                     temperature, seeds, request_ids, pos_base, accepted_len_out, out_tokens,
                     p_draft_out, row_stats_out, status, scratch, need, stream);
}
