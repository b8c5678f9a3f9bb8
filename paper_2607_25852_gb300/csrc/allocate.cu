// allocate.cu -- D-cut verification-depth allocation (Section 4.2 of arxiv
// 2607.25852) in one CTA on sm_103a.
//
// At most SPEC_MAX_ALLOC_POSITIONS = 8192 positions, so the whole problem fits
// in shared memory.  Every position (i, k) becomes one 64-bit key
//   bits(s_{i,k}) << 32 | (0xFFFF - k) << 16 | (0xFFFF - i)
// whose descending order is the allocator's total order: s >= 0, so the fp32
// bit pattern is monotone in s; then shallower k first (the paper's tie rule);
// then lower request index.  A bitonic network sorts the keys descending; an
// inclusive scan of floor(s * 2^40) over the sorted order gives every
// candidate's utility U(T) = prefix[T - 1] exactly, the first maximiser of
// U / cost is chosen, and the kept prefixes are packed densely.
#include <float.h>
#include <math.h>

#include <algorithm>

#include "spec_internal.cuh"

namespace spec {

constexpr int kAllocThreads = 1024;

__device__ __forceinline__ unsigned long long position_key(float s, int k, int i) {
  return ((unsigned long long)__float_as_uint(s) << 32) |
         ((unsigned long long)(0xFFFFu - (unsigned)k) << 16) | (unsigned long long)(0xFFFFu - (unsigned)i);
}

// Inclusive block scan of one int64 value per thread (kAllocThreads threads).
__device__ __forceinline__ long long block_inclusive_scan(long long x, long long* warp_tot) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
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
  const long long before = warp > 0 ? warp_tot[warp - 1] : 0;
  __syncthreads();  // warp_tot reusable after return
  return x + before;
}

__global__ void __launch_bounds__(kAllocThreads) allocate_kernel(const AllocLaunch p) {
  extern __shared__ unsigned long long smem[];
  unsigned long long* keys = smem;                                     // [npad]
  long long* prefix = reinterpret_cast<long long*>(smem + p.npad);     // [npad], later counts
  __shared__ long long warp_tot[32];
  __shared__ int sh_best_c;
  __shared__ int sh_bad;

  const int B = p.B, K = p.K, N = B * (K + 1), npad = p.npad;
  const int tid = threadIdx.x;
  if (tid == 0) sh_bad = 0;
  __syncthreads();

  // ---- Eq. (dcut-score): fp32 prefix products, one request per thread ----
  for (int i = tid; i < B; i += kAllocThreads) {
    float s = 1.0f;
    keys[i * (K + 1)] = position_key(s, 0, i);
    for (int k = 1; k <= K; ++k) {
      float c = p.conf[(size_t)i * K + (k - 1)];
      if (!(c >= 0.0f && c <= 1.0f)) {
        sh_bad = 1;
        c = 0.0f;
      }
      s = __fmul_rn(s, c);
      keys[i * (K + 1) + k] = position_key(s, k, i);
    }
  }
  for (int q = N + tid; q < npad; q += kAllocThreads) keys[q] = 0ull;  // sorts last
  __syncthreads();

  // ---- bitonic sort, descending ----
  for (int size = 2; size <= npad; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int t = tid; t < (npad >> 1); t += kAllocThreads) {
        const int lo = 2 * stride * (t / stride) + (t % stride);
        const int hi = lo + stride;
        const bool desc = (lo & size) == 0;
        const unsigned long long a = keys[lo], b = keys[hi];
        if ((a < b) == desc) {
          keys[lo] = b;
          keys[hi] = a;
        }
      }
      __syncthreads();
    }
  }

  // ---- inclusive scan of floor(s * 2^40) in sorted order ----
  const int per = (npad + kAllocThreads - 1) / kAllocThreads;
  const int q0 = tid * per;
  long long local = 0;
  for (int q = q0; q < q0 + per && q < npad; ++q) {
    const float s = __uint_as_float((unsigned)(keys[q] >> 32));
    local += q < N ? (long long)__float2ll_rd(s * 0x1p40f) : 0ll;
  }
  const long long incl = block_inclusive_scan(local, warp_tot);
  long long run = incl - local;
  for (int q = q0; q < q0 + per && q < npad; ++q) {
    const float s = __uint_as_float((unsigned)(keys[q] >> 32));
    run += q < N ? (long long)__float2ll_rd(s * 0x1p40f) : 0ll;
    prefix[q] = run;
  }
  __syncthreads();

  // ---- Eq. (dcut-select): first maximiser of U / cost ----
  if (tid == 0) {
    int best_c = 0;
    double best_obj = -INFINITY;
    for (int c = 0; c < p.M; ++c) {
      const double util = ldexp((double)prefix[p.cand_T[c] - 1], -40);
      if (p.utility_out) p.utility_out[c] = util;
      const double obj = util / p.cand_cost[c];
      if (obj > best_obj) {
        best_obj = obj;
        best_c = c;
      }
    }
    sh_best_c = best_c;
  }
  __syncthreads();
  const int T = p.cand_T[sh_best_c];

  // ---- keep depths: count the selected positions per request ----
  int* counts = reinterpret_cast<int*>(prefix);  // prefix no longer needed
  for (int i = tid; i < B; i += kAllocThreads) counts[i] = 0;
  __syncthreads();
  for (int q = tid; q < T; q += kAllocThreads) {
    const int i = 0xFFFF - (int)(keys[q] & 0xFFFFull);
    atomicAdd(&counts[i], 1);
  }
  __syncthreads();

  // ---- row offsets: exclusive scan of (n_i + 1) = counts ----
  const int perB = (B + kAllocThreads - 1) / kAllocThreads;
  const int b0 = tid * perB;
  long long lsum = 0;
  for (int i = b0; i < b0 + perB && i < B; ++i) lsum += counts[i];
  const long long bincl = block_inclusive_scan(lsum, warp_tot);
  long long off = bincl - lsum;
  int* offsets = reinterpret_cast<int*>(prefix) + B;  // [B+1] after counts
  for (int i = b0; i < b0 + perB && i < B; ++i) {
    offsets[i] = (int)off;
    p.row_offsets_out[i] = (int)off;
    p.depth_out[i] = counts[i] - 1;
    off += counts[i];
  }
  if (tid == kAllocThreads - 1) {
    p.row_offsets_out[B] = (int)bincl;
    *p.chosen_T_out = T;
  }
  __syncthreads();

  // ---- dense packing of the kept prefixes ----
  for (int q = tid; q < N; q += kAllocThreads) {
    if (q < T) {
      const unsigned long long key = keys[q];
      const int i = 0xFFFF - (int)(key & 0xFFFFull);
      const int k = 0xFFFF - (int)((key >> 16) & 0xFFFFull);
      const int row = offsets[i] + k;
      p.packed_tokens_out[row] = k == 0 ? p.last_tokens[i] : p.drafts[(size_t)i * K + (k - 1)];
      p.packed_pos_out[row] = p.pos_base[i] + k;
    } else {
      p.packed_tokens_out[q] = -1;
      p.packed_pos_out[q] = -1;
    }
  }
  if (tid == 0 && sh_bad) report(p.status, SPEC_ERR_BAD_INPUT);
}

cudaError_t launch_allocate(const AllocLaunch& p, cudaStream_t stream) {
  // keys [npad] u64, then one region reused for the prefix sums [npad] i64 and
  // for counts [B] + offsets [B+1] i32
  const size_t region = std::max((size_t)p.npad * 8, ((size_t)2 * p.B + 2) * 4);
  const size_t smem = (size_t)p.npad * 8 + ((region + 15) / 16) * 16;
  cudaError_t err = cudaFuncSetAttribute(allocate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
  if (err != cudaSuccess) return err;
  allocate_kernel<<<1, kAllocThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace spec
