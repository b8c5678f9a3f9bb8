// spec_internal.cuh -- device helpers and launch parameters shared by the
// kernels of libspec (sm_103a).  Nothing here is part of the public ABI.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>
#include <stdint.h>

#include "spec.h"

namespace spec {

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two 32x32
// multiplies whose high halves are mixed with the other counter words and the
// round key; the key advances by the two Weyl increments every round.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    const uint32_t hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo0 = 0xD2511F53u * c.x;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z);
    const uint32_t lo1 = 0xCD9E8D57u * c.z;
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return c;
}

// Counter of one draw (the layout documented in spec.h).
__device__ __forceinline__ uint4 draw_counter(uint32_t position, uint64_t request,
                                              uint32_t purpose, uint32_t sub) {
  return make_uint4(position, (uint32_t)request, (uint32_t)(request >> 32),
                    (purpose << 28) | sub);
}

// ---------------------------------------------------------------------------
// Status word: first error wins.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void report(int32_t* status, int code) {
  if (status) atomicCAS(reinterpret_cast<int*>(status), 0, code);
}

// ---------------------------------------------------------------------------
// Loads
// ---------------------------------------------------------------------------
// Streaming 16-byte load: read once, keep out of L1.
__device__ __forceinline__ uint4 ldg_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

template <typename T>
__device__ __forceinline__ float load_elem(const T* p);
template <>
__device__ __forceinline__ float load_elem<float>(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float load_elem<__nv_bfloat16>(const __nv_bfloat16* p) {
  const uint16_t bits = __ldg(reinterpret_cast<const unsigned short*>(p));
  return __uint_as_float(((uint32_t)bits) << 16);
}

__device__ __forceinline__ float load_any(const void* base, int dtype, int64_t idx) {
  return dtype == SPEC_F32 ? load_elem(static_cast<const float*>(base) + idx)
                           : load_elem(static_cast<const __nv_bfloat16*>(base) + idx);
}

// ---------------------------------------------------------------------------
// Programmatic dependent launch
// ---------------------------------------------------------------------------
// Programmatic dependent launch: let the next kernel on the stream start
// launching / wait until the previous kernel has completed and flushed.
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait_prerequisites() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// An NVTX range over one host call (the library's entry points), for
// Nsight timelines.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
};

// Launch `kernel` so that it may start while the previous kernel on the
// stream drains (programmatic stream serialization).  Every kernel launched
// this way calls pdl_wait_prerequisites() before it reads anything that an
// earlier kernel writes, so the overlap covers launch latency only.
template <typename... Args>
inline cudaError_t launch_after_previous(void (*kernel)(Args...), dim3 grid, dim3 block, size_t smem,
                                         cudaStream_t stream, Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// max with NaN propagation (PTX max.NaN)
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float d;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
  return d;
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ---------------------------------------------------------------------------
// Workspace records
// ---------------------------------------------------------------------------
// Per (row, vocabulary chunk) partial of the streaming pass.
//   softmax: m = max logit, s = sum_v 2^(l_v*c2 - fl(m*c2)), flags bit0 = NaN/+inf seen
//   greedy : m = max logit, idx = lowest index attaining it, flags bit0 = NaN seen
struct alignas(16) RowPartial {
  float m;
  float s;
  int32_t idx;
  int32_t flags;
};

// A partial written by another CTA of the same kernel: read at L2 (.cg).
__device__ __forceinline__ RowPartial load_partial_cg(const RowPartial* ptr) {
  const uint4 v = __ldcg(reinterpret_cast<const uint4*>(ptr));
  RowPartial r;
  r.m = __uint_as_float(v.x);
  r.s = __uint_as_float(v.y);
  r.idx = (int32_t)v.z;
  r.flags = (int32_t)v.w;
  return r;
}

// Per (request, vocabulary chunk) partial of the sampling pass: the best key
// and index of the residual race (weights max(0, p - q)) and of the race on p.
struct alignas(16) RacePartial {
  float key_r;
  int32_t idx_r;
  float key_p;
  int32_t idx_p;
};

// Per request, written by its decision for the sampling pass (t > 0).
struct alignas(16) ReqRec {
  int32_t a;          // accepted drafts; the sampled row is the request's row a
  int32_t flags;      // bit0 bad input, bit1 a draft was rejected, bit2 residual against a dense q row
  int32_t z_excl;     // the rejected draft token with one-hot q (excluded from the race), else -1
  uint32_t position;  // pos_base + a: the Philox position of the sampled token
  int64_t srow;       // packed row index of the sampled row
  float M2;           // fl(max * c2) of the sampled row
  float invS;         // 1 / S of the sampled row
};

// ---------------------------------------------------------------------------
// Launch parameters
// ---------------------------------------------------------------------------
struct VerifyLaunch {
  const void* logits;
  int logits_dtype;
  const int32_t* row_offsets;
  const int32_t* depth;
  const int32_t* drafts;
  const void* q;
  int q_dtype;
  bool dense_q;         // q given (t > 0): residual draws against it
  int B, K, V;
  float temperature;
  float c2;            // log2(e) / t  (0 when t == 0)
  float inv_t;         // 1 / t
  const uint64_t* seeds;
  const uint64_t* request_ids;
  const int64_t* pos_base;
  int32_t* accepted_len;
  int32_t* out_tokens;
  float* p_draft;
  float* row_stats;
  int32_t* status;
  // workspace carve-up
  RowPartial* row_part;   // [R_max * NC]
  RacePartial* race_part; // [B * NCS]
  float2* draft_view;     // [R_max]: (logit, q) at each row's draft token (t > 0)
  uint32_t* counters;     // [B] sampling-pass arrivals per request
  int R_max;              // B * (K + 1)
  int NC;                 // vocabulary chunks per row, streaming pass
  int chunk;              // elements per chunk (multiple of 8)
  int NCS;                // vocabulary chunks per request, sampling pass
  int chunk_s;            // elements per sampling chunk (multiple of 8)
  bool vec_s;             // sampling pass may use 16-byte loads
};

struct AllocLaunch {
  const float* conf;
  int B, K, M;
  int32_t cand_T[SPEC_MAX_CANDIDATES];
  double cand_cost[SPEC_MAX_CANDIDATES];
  const int32_t* last_tokens;
  const int32_t* drafts;
  const int64_t* pos_base;
  int32_t* depth_out;
  int32_t* row_offsets_out;
  int32_t* packed_tokens_out;
  int64_t* packed_pos_out;
  int32_t* chosen_T_out;
  double* utility_out;
  int32_t* status;
  int npad;  // next power of two >= B(K+1)
};

struct CommitLaunch {
  const int32_t* accepted_len;
  const int32_t* out_tokens;
  const int32_t* row_offsets;
  const void* hidden;
  int64_t row_bytes;
  int B, K;
  int32_t* packed_tokens_out;
  int32_t* commit_offsets_out;
  void* hidden_out;
  int32_t* status;
};

// Workspace geometry (device independent).
struct VerifyGeometry {
  int NC, chunk, NCS, chunk_s;
  size_t row_part_off, race_part_off, view_off, counters_off, bytes;  // [counters_off, bytes) starts at zero
};
VerifyGeometry verify_geometry(int B, int K, int V);

// Launchers (return cudaSuccess or the launch error).
cudaError_t launch_verify(const VerifyLaunch& p, cudaStream_t stream, cudaEvent_t ev_before,
                          cudaEvent_t ev_after);
cudaError_t launch_allocate(const AllocLaunch& p, cudaStream_t stream);
cudaError_t launch_commit(const CommitLaunch& p, cudaStream_t stream);

// spec_verify's host checks and launches, with an optional hook that runs
// after every check has passed and before anything is launched.
int verify_impl(const void* logits, int logits_dtype, const int32_t* row_offsets, const int32_t* depth,
                const int32_t* draft_tokens, const void* q, int q_dtype, int B, int K, int V, float temperature,
                const uint64_t* seeds, const uint64_t* request_ids, const int64_t* pos_base,
                int32_t* accepted_len_out, int32_t* out_tokens, float* p_draft_out, float* row_stats_out,
                int32_t* status, void* ws, size_t ws_bytes, cudaStream_t stream,
                cudaError_t (*pre_launch)(void*, cudaStream_t), void* hook_ctx);

}  // namespace spec
