// abi.cu -- extern "C" entry points of libspec (declared in include/spec.h).
//
// Host side only: argument checks, workspace carve-up and kernel launches.
// Nothing here allocates device memory, synchronises a stream or reads device
// memory, so every entry point is stream-ordered.
#include <math.h>
#include <stdint.h>

#include "spec_internal.cuh"

namespace {

using spec::NvtxRange;

cudaEvent_t g_profile_before = nullptr;
cudaEvent_t g_profile_after = nullptr;

int next_pow2(int x) {
  int p = 1;
  while (p < x) p <<= 1;
  return p;
}

bool verify_shape_ok(int B, int K, int V) {
  if (B < 1 || K < 0 || K > SPEC_MAX_DRAFTS || V < 1 || V >= SPEC_MAX_VOCAB) return false;
  const long long R = (long long)B * (K + 1);
  return R <= (1LL << 28);
}

bool dtype_ok(int dt) { return dt == SPEC_BF16 || dt == SPEC_F32; }

}  // namespace

extern "C" {

const char* spec_error_string(int code) {
  switch (code) {
    case SPEC_OK: return "ok";
    case SPEC_ERR_INVALID_ARG: return "invalid argument";
    case SPEC_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case SPEC_ERR_CUDA: return "CUDA runtime error";
    case SPEC_ERR_BAD_INPUT: return "bad input data detected on the device";
    case SPEC_ERR_TIMEOUT: return "bounded device wait timed out";
    case SPEC_ERR_TOO_LARGE: return "shape needs more scratch than the static buffer holds";
    default: return "unknown error code";
  }
}

int spec_version(void) { return SPEC_ABI_VERSION; }

int spec_pointer_device_readable(const void* ptr) {
  if (!ptr) return 0;
  cudaPointerAttributes a{};
  if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
    cudaGetLastError();  // clear the error this query may leave
    return 0;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return 1;
  return a.type == cudaMemoryTypeHost && a.devicePointer == ptr ? 1 : 0;
}

int spec_budget_from_ratios(int B, int K, const int32_t* num, const int32_t* den, int M,
                            int32_t* cand_T_out) {
  if (B < 1 || K < 0 || M < 1 || !num || !den || !cand_T_out) return SPEC_ERR_INVALID_ARG;
  const long long full = (long long)B * (K + 1);
  for (int m = 0; m < M; ++m) {
    if (den[m] <= 0 || num[m] < 0 || num[m] > den[m]) return SPEC_ERR_INVALID_ARG;
  }
  for (int m = 0; m < M; ++m) {
    long long T = ((long long)num[m] * full + den[m] - 1) / den[m];  // ceil(rho * B(K+1))
    if (T < B) T = B;                                                // Eq. (dcut-budget): max(B, .)
    cand_T_out[m] = (int32_t)T;
  }
  return SPEC_OK;
}

size_t spec_allocate_workspace(int, int, int) { return 0; }

int spec_allocate(const float* conf, int B, int K, const int32_t* cand_T, const double* cand_cost,
                  int M, const int32_t* last_tokens, const int32_t* draft_tokens,
                  const int64_t* pos_base, int32_t* depth_out, int32_t* row_offsets_out,
                  int32_t* packed_tokens_out, int64_t* packed_pos_out, int32_t* chosen_T_out,
                  double* utility_out, int32_t* status, void* ws, size_t ws_bytes,
                  cudaStream_t stream) {
  (void)ws;
  (void)ws_bytes;
  NvtxRange range("spec_allocate");
  if (B < 1 || K < 0 || K > SPEC_MAX_DRAFTS || M < 1 || M > SPEC_MAX_CANDIDATES)
    return SPEC_ERR_INVALID_ARG;
  const long long N = (long long)B * (K + 1);
  if (N > SPEC_MAX_ALLOC_POSITIONS) return SPEC_ERR_INVALID_ARG;
  if ((K > 0 && (!conf || !draft_tokens)) || !cand_T || !cand_cost || !last_tokens || !pos_base ||
      !depth_out || !row_offsets_out || !packed_tokens_out || !packed_pos_out || !chosen_T_out)
    return SPEC_ERR_INVALID_ARG;
  spec::AllocLaunch p{};
  for (int m = 0; m < M; ++m) {
    if (cand_T[m] < B || cand_T[m] > N) return SPEC_ERR_INVALID_ARG;
    if (!(cand_cost[m] > 0.0) || isinf(cand_cost[m])) return SPEC_ERR_INVALID_ARG;
    p.cand_T[m] = cand_T[m];
    p.cand_cost[m] = cand_cost[m];
  }
  p.conf = conf;
  p.B = B;
  p.K = K;
  p.M = M;
  p.last_tokens = last_tokens;
  p.drafts = draft_tokens;
  p.pos_base = pos_base;
  p.depth_out = depth_out;
  p.row_offsets_out = row_offsets_out;
  p.packed_tokens_out = packed_tokens_out;
  p.packed_pos_out = packed_pos_out;
  p.chosen_T_out = chosen_T_out;
  p.utility_out = utility_out;
  p.status = status;
  p.npad = next_pow2((int)N);
  return spec::launch_allocate(p, stream) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

size_t spec_verify_workspace(int B, int K, int V) {
  if (!verify_shape_ok(B, K, V)) return 0;
  return spec::verify_geometry(B, K, V).bytes;
}

int spec_verify(const void* logits, int logits_dtype, const int32_t* row_offsets,
                const int32_t* depth, const int32_t* draft_tokens, const void* q, int q_dtype,
                int B, int K, int V, float temperature, const uint64_t* seeds,
                const uint64_t* request_ids, const int64_t* pos_base, int32_t* accepted_len_out,
                int32_t* out_tokens, float* p_draft_out, float* row_stats_out, int32_t* status,
                void* ws, size_t ws_bytes, cudaStream_t stream) {
  return spec::verify_impl(logits, logits_dtype, row_offsets, depth, draft_tokens, q, q_dtype, B, K, V,
                           temperature, seeds, request_ids, pos_base, accepted_len_out, out_tokens,
                           p_draft_out, row_stats_out, status, ws, ws_bytes, stream, nullptr, nullptr);
}

}  // extern "C"

// spec_verify with a hook that runs once every host-side check has passed,
// immediately before the first launch (nullptr: none).  A hook that fails
// makes the call return SPEC_ERR_CUDA with nothing launched.
int spec::verify_impl(const void* logits, int logits_dtype, const int32_t* row_offsets, const int32_t* depth,
                      const int32_t* draft_tokens, const void* q, int q_dtype, int B, int K, int V,
                      float temperature, const uint64_t* seeds, const uint64_t* request_ids,
                      const int64_t* pos_base, int32_t* accepted_len_out, int32_t* out_tokens,
                      float* p_draft_out, float* row_stats_out, int32_t* status, void* ws, size_t ws_bytes,
                      cudaStream_t stream, cudaError_t (*pre_launch)(void*, cudaStream_t), void* hook_ctx) {
  NvtxRange range("spec_verify");
  cudaEvent_t ev_before = g_profile_before, ev_after = g_profile_after;
  g_profile_before = g_profile_after = nullptr;
  if (!verify_shape_ok(B, K, V) || !dtype_ok(logits_dtype)) return SPEC_ERR_INVALID_ARG;
  if (!(temperature >= 0.0f) || isinf(temperature)) return SPEC_ERR_INVALID_ARG;
  if (q && !dtype_ok(q_dtype)) return SPEC_ERR_INVALID_ARG;
  if (!logits || (K > 0 && !draft_tokens) || !seeds || !request_ids || !pos_base ||
      !accepted_len_out || !out_tokens)
    return SPEC_ERR_INVALID_ARG;
  const spec::VerifyGeometry g = spec::verify_geometry(B, K, V);
  if (!ws || ws_bytes < g.bytes || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return SPEC_ERR_WORKSPACE;
  if (row_stats_out && (reinterpret_cast<uintptr_t>(row_stats_out) & 7u) != 0)
    return SPEC_ERR_INVALID_ARG;

  spec::VerifyLaunch p{};
  p.logits = logits;
  p.logits_dtype = logits_dtype;
  p.row_offsets = row_offsets;
  p.depth = depth;
  p.drafts = draft_tokens;
  p.q = temperature > 0.0f ? q : nullptr;
  p.dense_q = p.q != nullptr;
  p.q_dtype = q_dtype;
  p.B = B;
  p.K = K;
  p.V = V;
  p.temperature = temperature;
  p.c2 = temperature > 0.0f ? (float)(1.4426950408889634 / (double)temperature) : 0.0f;
  p.inv_t = temperature > 0.0f ? (float)(1.0 / (double)temperature) : 0.0f;
  p.seeds = seeds;
  p.request_ids = request_ids;
  p.pos_base = pos_base;
  p.accepted_len = accepted_len_out;
  p.out_tokens = out_tokens;
  p.p_draft = p_draft_out;
  p.row_stats = row_stats_out;
  p.status = status;
  char* base = static_cast<char*>(ws);
  p.row_part = reinterpret_cast<spec::RowPartial*>(base + g.row_part_off);
  p.race_part = reinterpret_cast<spec::RacePartial*>(base + g.race_part_off);
  p.draft_view = reinterpret_cast<float2*>(base + g.view_off);
  p.counters = reinterpret_cast<uint32_t*>(base + g.counters_off);
  p.R_max = B * (K + 1);
  p.NC = g.NC;
  p.chunk = g.chunk;
  p.NCS = g.NCS;
  p.chunk_s = g.chunk_s;
  {
    // 16-byte loads in the sampling pass: V a multiple of 8 (every chunk
    // starts on a group of 8) and both row bases 16-byte aligned.
    const size_t esize = logits_dtype == SPEC_F32 ? 4 : 2, qsize = q_dtype == SPEC_F32 ? 4 : 2;
    const bool q_ok = p.q == nullptr || (reinterpret_cast<uintptr_t>(p.q) % 16 == 0 && (V * qsize) % 16 == 0);
    p.vec_s = V % 8 == 0 && reinterpret_cast<uintptr_t>(logits) % 16 == 0 && (V * esize) % 16 == 0 && q_ok;
  }
  if (pre_launch && pre_launch(hook_ctx, stream) != cudaSuccess) return SPEC_ERR_CUDA;
  return spec::launch_verify(p, stream, ev_before, ev_after) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

extern "C" {

int spec_commit(const int32_t* accepted_len, const int32_t* out_tokens, const int32_t* row_offsets,
                const void* hidden, int hidden_dtype, int B, int K, int H,
                int32_t* packed_tokens_out, int32_t* commit_offsets_out, void* hidden_out,
                int32_t* status, cudaStream_t stream) {
  NvtxRange range("spec_commit");
  if (B < 1 || K < 0 || K > SPEC_MAX_DRAFTS || (long long)B * (K + 1) > (1LL << 28))
    return SPEC_ERR_INVALID_ARG;
  if (!accepted_len || !out_tokens || !packed_tokens_out || !commit_offsets_out)
    return SPEC_ERR_INVALID_ARG;
  if ((hidden != nullptr) != (hidden_out != nullptr)) return SPEC_ERR_INVALID_ARG;
  if (hidden && (!dtype_ok(hidden_dtype) || H < 1)) return SPEC_ERR_INVALID_ARG;
  spec::CommitLaunch p{};
  p.accepted_len = accepted_len;
  p.out_tokens = out_tokens;
  p.row_offsets = row_offsets;
  p.hidden = hidden;
  p.row_bytes = hidden ? (int64_t)H * (hidden_dtype == SPEC_F32 ? 4 : 2) : 0;
  p.B = B;
  p.K = K;
  p.packed_tokens_out = packed_tokens_out;
  p.commit_offsets_out = commit_offsets_out;
  p.hidden_out = hidden_out;
  p.status = status;
  return spec::launch_commit(p, stream) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

int spec_profile_stream_pass(cudaEvent_t before, cudaEvent_t after) {
  if ((before == nullptr) != (after == nullptr)) return SPEC_ERR_INVALID_ARG;
  g_profile_before = before;
  g_profile_after = after;
  return SPEC_OK;
}

}  // extern "C"
