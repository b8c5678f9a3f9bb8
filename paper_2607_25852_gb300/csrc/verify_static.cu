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
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "spec_internal.cuh"

namespace {

// The scratch itself.  Zero at module load; each call clears the part that
// must start at zero.
static __device__ __align__(256) unsigned char g_verify_scratch[SPEC_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 256;
std::mutex g_setup_mutex;
struct ScratchSlot {
  CUcontext ctx;  // the context the address belongs to
  void* ptr;
};
ScratchSlot g_scratch[kMaxDevices] = {};

// cuCtxGetCurrent through the runtime's driver entry-point query (the library
// does not link the driver API).
PFN_cuCtxGetCurrent_v4000 ctx_getter() {
  static PFN_cuCtxGetCurrent_v4000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &ptr, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(ptr);
  }
  return fn;
}

// Device address of g_verify_scratch on the current device.  In host code the
// name g_verify_scratch only denotes a host-side stand-in, so the address is
// looked up with the device current and cached, once per device and context:
// a new context on the device (after cudaDeviceReset, say) loads the module
// again, possibly at another address, and is looked up afresh.
int scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SPEC_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  // cudaGetSymbolAddress makes the device's primary context current if none
  // is; the context is read after it.
  void* ptr = g_scratch[dev].ptr;
  CUcontext ctx = nullptr;
  auto get_ctx = ctx_getter();
  if (ptr != nullptr && get_ctx && get_ctx(&ctx) == CUDA_SUCCESS && ctx == g_scratch[dev].ctx) {
    *out = ptr;
    return SPEC_OK;
  }
  ptr = nullptr;
  if (cudaGetSymbolAddress(&ptr, g_verify_scratch) != cudaSuccess || ptr == nullptr) return SPEC_ERR_CUDA;
  ctx = nullptr;
  if (get_ctx && get_ctx(&ctx) == CUDA_SUCCESS && ctx != nullptr) g_scratch[dev] = ScratchSlot{ctx, ptr};
  else g_scratch[dev] = ScratchSlot{nullptr, nullptr};  // no context to key on: look up every call
  *out = ptr;
  return SPEC_OK;
}

// The part of the scratch that must start at zero (the arrival counters),
// cleared on the call's stream once every argument check has passed.
struct ClearRange {
  void* ptr;
  size_t bytes;
};
cudaError_t clear_counters(void* ctx, cudaStream_t stream) {
  const ClearRange* r = static_cast<const ClearRange*>(ctx);
  return cudaMemsetAsync(r->ptr, 0, r->bytes, stream);
}

}  // namespace

extern "C" int spec_verify_static(const void* logits, int logits_dtype, const int32_t* row_offsets,
                                  const int32_t* depth, const int32_t* draft_tokens, const void* q,
                                  int q_dtype, int B, int K, int V, float temperature,
                                  const uint64_t* seeds, const uint64_t* request_ids,
                                  const int64_t* pos_base, int32_t* accepted_len_out,
                                  int32_t* out_tokens, float* p_draft_out, float* row_stats_out,
                                  int32_t* status, cudaStream_t stream) {
  spec::NvtxRange range("spec_verify_static");
  const size_t need = spec_verify_workspace(B, K, V);
  if (need == 0) return SPEC_ERR_INVALID_ARG;
  if (need > (size_t)SPEC_STATIC_SCRATCH_BYTES) return SPEC_ERR_TOO_LARGE;
  void* scratch = nullptr;
  const int rc = scratch_address(&scratch);
  if (rc != SPEC_OK) return rc;
  // The arrival counters must be zero when a call starts; clear them rather
  // than rely on what the previous call left behind.  The clear is queued
  // only after spec_verify's argument checks, so a rejected call leaves the
  // stream and the scratch untouched.
  const spec::VerifyGeometry g = spec::verify_geometry(B, K, V);
  ClearRange clear{static_cast<char*>(scratch) + g.counters_off, need - g.counters_off};
  return spec::verify_impl(logits, logits_dtype, row_offsets, depth, draft_tokens, q, q_dtype, B, K, V,
                           temperature, seeds, request_ids, pos_base, accepted_len_out, out_tokens, p_draft_out,
                           row_stats_out, status, scratch, need, stream, clear_counters, &clear);
}
