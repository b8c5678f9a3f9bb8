// commit.cu -- pack the committed round for the drafter's next step
// (arxiv 2607.25852, Section 1: the verified prefix plus one target token is
// committed; Sections 3.1 and 6: the drafter conditions on the target hidden
// states of the committed positions).
//
// One CTA per (request, row j <= a_i): it writes token j of the request at
// commit_offsets[i] + j and copies hidden row row_offsets[i] + j there with
// 16-byte loads and stores.  commit_offsets[i] = sum_{i' < i} (a_{i'} + 1) is
// summed by the CTA itself for small batches, or produced first by a one-CTA
// scan kernel into commit_offsets_out for large ones.
#include "spec_internal.cuh"

namespace spec {

constexpr int kCommitThreads = 256;
constexpr int kScanThreads = 1024;
constexpr int kInlineScanMaxB = 256;

__device__ __forceinline__ int committed_len(const CommitLaunch& p, int i) {
  const int a = p.accepted_len[i];
  return (a >= 0 && a <= p.K) ? a : 0;  // out-of-range lengths count as 0 (reported)
}

__global__ void __launch_bounds__(kScanThreads) commit_scan_kernel(const CommitLaunch p) {
  __shared__ long long warp_tot[32];
  __shared__ long long carry;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  pdl_wait_prerequisites();  // accepted lengths come from the verification
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < p.B; base += kScanThreads) {
    const int i = base + threadIdx.x;
    long long x = i < p.B ? (long long)committed_len(p, i) + 1 : 0;
    const long long mine = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xFFFFFFFFu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    if (warp == 0) {
      long long t = warp_tot[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xFFFFFFFFu, t, o);
        if (lane >= o) t += y;
      }
      warp_tot[lane] = t;
    }
    __syncthreads();
    const long long incl = x + (warp > 0 ? warp_tot[warp - 1] : 0) + carry;
    if (i < p.B) p.commit_offsets_out[i] = (int32_t)(incl - mine);
    __syncthreads();
    if (threadIdx.x == kScanThreads - 1) carry = incl;
    __syncthreads();
  }
  if (threadIdx.x == 0) p.commit_offsets_out[p.B] = (int32_t)carry;
}

template <bool kScanned>
__global__ void __launch_bounds__(kCommitThreads) commit_kernel(const CommitLaunch p) {
  const int K1 = p.K + 1;
  const int i = blockIdx.x / K1;
  const int j = blockIdx.x - i * K1;
  pdl_wait_prerequisites();  // accepted lengths and tokens come from the verification
  // ---- one round trip: this request's length and row, every length before
  // it (inline offsets), and the token ----
  const int a_raw = p.accepted_len[i];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int before = 0;
  if (!kScanned && (int)threadIdx.x < i) before = committed_len(p, threadIdx.x) + 1;
  const long long row_i = p.row_offsets ? (long long)p.row_offsets[i] : (long long)i * K1;
  const long long R = p.row_offsets ? (long long)p.row_offsets[p.B] : (long long)p.B * K1;
  const int32_t token = threadIdx.x == 0 ? p.out_tokens[(size_t)i * K1 + j] : 0;
  const int a = (a_raw >= 0 && a_raw <= p.K) ? a_raw : 0;  // out-of-range lengths count as 0 (reported)
  if (j == 0 && threadIdx.x == 0 && a != a_raw) report(p.status, SPEC_ERR_BAD_INPUT);
  if (j > a) return;

  __shared__ int sh_off;
  if (kScanned) {
    if (threadIdx.x == 0) sh_off = p.commit_offsets_out[i];
  } else {
    // sum_{i' < i} (a_{i'} + 1); i < kInlineScanMaxB <= kCommitThreads
    __shared__ int warp_sum[kCommitThreads / 32];
    int x = before;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
    if (lane == 0) warp_sum[warp] = x;
    __syncthreads();
    if (threadIdx.x == 0) {
      int s = 0;
      for (int w = 0; w < kCommitThreads / 32; ++w) s += warp_sum[w];
      sh_off = s;
      if (j == 0) {
        p.commit_offsets_out[i] = s;
        if (i == p.B - 1) p.commit_offsets_out[p.B] = s + a + 1;
      }
    }
  }
  __syncthreads();
  const int dst = sh_off + j;
  if (threadIdx.x == 0) p.packed_tokens_out[dst] = token;
  if (p.hidden == nullptr || p.hidden_out == nullptr) return;

  const long long src_row = row_i + j;
  if (src_row < 0 || src_row >= R) {
    if (threadIdx.x == 0) report(p.status, SPEC_ERR_BAD_INPUT);
    return;
  }
  const char* src = static_cast<const char*>(p.hidden) + src_row * p.row_bytes;
  char* out = static_cast<char*>(p.hidden_out) + (long long)dst * p.row_bytes;
  const bool aligned = ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(out) |
                         (uintptr_t)p.row_bytes) & 15u) == 0;
  if (aligned) {
    const uint4* s4 = reinterpret_cast<const uint4*>(src);
    uint4* d4 = reinterpret_cast<uint4*>(out);
    const int n4 = (int)(p.row_bytes >> 4);
    for (int k = threadIdx.x; k < n4; k += kCommitThreads) d4[k] = ldg_stream(s4 + k);
  } else {
    for (long long k = threadIdx.x; k < p.row_bytes; k += kCommitThreads) out[k] = src[k];
  }
}

cudaError_t launch_commit(const CommitLaunch& p, cudaStream_t stream) {
  const unsigned grid = (unsigned)((long long)p.B * (p.K + 1));
  cudaError_t err;
  if (p.B <= kInlineScanMaxB) {
    err = launch_after_previous(commit_kernel<false>, dim3(grid), dim3(kCommitThreads), 0, stream, p);
  } else {
    err = launch_after_previous(commit_scan_kernel, dim3(1), dim3(kScanThreads), 0, stream, p);
    if (err != cudaSuccess) return err;
    err = launch_after_previous(commit_kernel<true>, dim3(grid), dim3(kCommitThreads), 0, stream, p);
  }
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

}  // namespace spec
