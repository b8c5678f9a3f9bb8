// allocate.cu -- D-cut verification-depth allocation (Section 4.2 of arxiv
// 2607.25852) in one CTA on sm_103a.
//
// At most SPEC_MAX_ALLOC_POSITIONS = 8192 positions, so the whole problem fits
// in shared memory.  Every position (i, k) becomes one 64-bit key
//   bits(s_{i,k}) << 32 | (0xFFFF - k) << 16 | (0xFFFF - i)
// whose descending order is the allocator's total order: s >= +0 (a -0
// confidence is taken as +0), so the fp32 bit pattern is monotone in s; then
// shallower k first (the paper's tie rule);
// then lower request index.  Keys are unique.
//
// Batches of at most 1024 requests and 1024 draft positions take
// allocate_small_kernel (below), which sorts the draft keys alone: a merge
// tree over the per-request runs padded to a power of two when they fit in
// 1024 slots, else a bitonic sort.  Larger batches take allocate_kernel:
// because s_{i,k} is non-increasing in k, each request's K+1 keys already form
// a run sorted in descending order.  A merge tree of ceil(log2 B) levels sorts
// the B runs: at every level each key finds its place in the merged pair by
// one binary search in the partner run.  An inclusive scan of floor(s * 2^40)
// in sorted order then gives every candidate's utility U(T) = prefix[T - 1]
// exactly; the first maximiser of U / cost is chosen and the kept prefixes
// are packed densely.
#include <float.h>
#include <limits.h>
#include <math.h>

#include <algorithm>
#include <atomic>

#include "spec_internal.cuh"

namespace spec {

constexpr int kAllocThreads = 1024;

__device__ __forceinline__ unsigned long long position_key(float s, int k, int i) {
  return ((unsigned long long)__float_as_uint(s) << 32) |
         ((unsigned long long)(0xFFFFu - (unsigned)k) << 16) | (unsigned long long)(0xFFFFu - (unsigned)i);
}

__device__ __forceinline__ unsigned long long lds_u64(uint32_t addr) {
  unsigned long long v;
  asm volatile("ld.shared.u64 %0, [%1];" : "=l"(v) : "r"(addr));
  return v;
}
__device__ __forceinline__ void sts_u64(uint32_t addr, unsigned long long v) {
  asm volatile("st.shared.u64 [%0], %1;" ::"r"(addr), "l"(v) : "memory");
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

// Shared-memory layout (dynamic): two key buffers of N entries, then
// pos_base [B] int64, the confidences [B][K] fp32 at the odd row stride K | 1
// (so that the threads of a warp, one request each, read distinct banks), the
// draft tokens [B*K] int32 and last_tokens [B] int32.
struct AllocSmem {
  unsigned long long* keys[2];
  float* conf;
  int32_t* drafts;
  int32_t* last;
  long long* pos;
};

__device__ __forceinline__ AllocSmem carve(unsigned char* base, int N, int BK, int B) {
  AllocSmem s;
  s.keys[0] = reinterpret_cast<unsigned long long*>(base);
  s.keys[1] = s.keys[0] + N;
  unsigned char* p = reinterpret_cast<unsigned char*>(s.keys[1] + N);
  s.pos = reinterpret_cast<long long*>(p);
  p += (size_t)B * 8;
  s.conf = reinterpret_cast<float*>(p);
  p += BK > 0 ? (size_t)(BK + B) * 4 : 0;
  s.drafts = reinterpret_cast<int32_t*>(p);
  p += (size_t)BK * 4;
  s.last = reinterpret_cast<int32_t*>(p);
  return s;
}

size_t allocate_smem_bytes(int B, int K) {
  const size_t N = (size_t)B * (K + 1), BK = (size_t)B * K;
  // at most 24 N + 8 B + 16 bytes <= 229,392 for N <= 8192 (K = 0 needs no
  // confidences: 16 N + 12 B + 16)
  return N * 16 + (size_t)B * 8 + (BK > 0 ? (BK + B) * 4 : 0) + BK * 4 + (size_t)B * 4 + 16;
}

__global__ void __launch_bounds__(kAllocThreads) allocate_kernel(const AllocLaunch p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int B = p.B, K = p.K, N = B * (K + 1), BK = B * K, L0 = K + 1;
  const int CS = K | 1;  // odd row stride of the staged confidences
  const AllocSmem sm = carve(smem_raw, N, BK, B);
  __shared__ long long warp_tot[32];
  __shared__ int sh_best_c;
  __shared__ int sh_bad;
  const int tid = threadIdx.x;
  if (tid == 0) sh_bad = 0;
  // The next kernel (the streaming pass) may launch now: it waits for this
  // one's completion before it reads the depths and row offsets.
  pdl_launch_dependents();
  // This kernel starts while the previous one on the stream drains; it reads
  // its inputs, and overwrites the arrays the previous round's kernels read,
  // only once that kernel has completed.
  pdl_wait_prerequisites();

  // ---- every global input in one round trip, coalesced ----
  for (int q = tid; q < BK; q += kAllocThreads) {
    const int i = q / K;
    sm.conf[q + i * (CS - K)] = p.conf[q];  // [i][k] at i * CS + k
    sm.drafts[q] = p.drafts[q];
  }
  for (int i = tid; i < B; i += kAllocThreads) {
    sm.last[i] = p.last_tokens[i];
    sm.pos[i] = p.pos_base[i];
  }
  __syncthreads();

  // ---- Eq. (dcut-score): fp32 prefix products; run i holds request i ----
  for (int i = tid; i < B; i += kAllocThreads) {
    float s = 1.0f;
    sm.keys[0][i * L0] = position_key(s, 0, i);
    for (int k = 1; k <= K; ++k) {
      float c = sm.conf[i * CS + (k - 1)];
      if (!(c >= 0.0f && c <= 1.0f)) {
        sh_bad = 1;
        c = 0.0f;
      }
      // -0 passes the range check and equals 0, but its sign bit would put
      // its key above every positive score: -0 + 0 = +0 drops the sign.
      c = __fadd_rn(c, 0.0f);
      s = __fmul_rn(s, c);
      sm.keys[0][i * L0 + k] = position_key(s, k, i);
    }
  }
  __syncthreads();

  // ---- merge tree over the B sorted runs (descending) ----
  // Level l merges runs of L = L0 * 2^l keys; position e lies in run
  // (e / L0) >> l.  N <= 8192, so 32-bit indices suffice.
  // The two key buffers by their shared-window addresses, so that every
  // probe of the searches is a shared-memory load (ld.shared).
  const uint32_t kbuf0 = (uint32_t)__cvta_generic_to_shared(sm.keys[0]);
  const uint32_t kbuf1 = (uint32_t)__cvta_generic_to_shared(sm.keys[1]);
  int cur = 0;
  for (int lev = 0, L = L0; L < N; ++lev, L *= 2) {
    const uint32_t in = cur ? kbuf1 : kbuf0, out = cur ? kbuf0 : kbuf1;
    for (int e = tid; e < N; e += kAllocThreads) {
      const int run = (e / L0) >> lev;
      const int start = run * L;
      const int pstart = (run ^ 1) * L;
      const unsigned long long x = lds_u64(in + 8u * (uint32_t)e);
      if (pstart >= N) {  // unpaired last run: copied through
        sts_u64(out + 8u * (uint32_t)e, x);
        continue;
      }
      const int plen = min(N, pstart + L) - pstart;
      // number of partner keys greater than x (the partner run is descending)
      int lo = 0, hi = plen;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (lds_u64(in + 8u * (uint32_t)(pstart + mid)) > x) lo = mid + 1;
        else hi = mid;
      }
      sts_u64(out + 8u * (uint32_t)(min(start, pstart) + (e - start) + lo), x);
    }
    __syncthreads();
    cur ^= 1;
  }
  const unsigned long long* keys = sm.keys[cur];
  long long* prefix = reinterpret_cast<long long*>(sm.keys[cur ^ 1]);  // free buffer

  // ---- inclusive scan of floor(s * 2^40) in sorted order ----
  const int per = (N + kAllocThreads - 1) / kAllocThreads;
  const int q0 = tid * per;
  long long local = 0;
  for (int q = q0; q < q0 + per && q < N; ++q)
    local += (long long)__float2ll_rd(__uint_as_float((unsigned)(keys[q] >> 32)) * 0x1p40f);
  const long long incl = block_inclusive_scan(local, warp_tot);
  long long run = incl - local;
  for (int q = q0; q < q0 + per && q < N; ++q) {
    run += (long long)__float2ll_rd(__uint_as_float((unsigned)(keys[q] >> 32)) * 0x1p40f);
    prefix[q] = run;
  }
  __syncthreads();

  // ---- Eq. (dcut-select): first maximiser of U / cost ----
  if (tid < 32) {
    // one lane per candidate (M <= 64: two per lane); the first maximiser
    // in candidate order wins ties, as a sequential scan would
    double best_obj = -INFINITY;
    int best_c = INT_MAX;
    for (int c = tid; c < p.M; c += 32) {
      const double U = ldexp((double)prefix[p.cand_T[c] - 1], -40);
      if (p.utility_out) p.utility_out[c] = U;
      const double obj = U / p.cand_cost[c];
      if (obj > best_obj) {  // c increases along the lane's loop
        best_obj = obj;
        best_c = c;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const double ob = __shfl_xor_sync(0xFFFFFFFFu, best_obj, o);
      const int cb = __shfl_xor_sync(0xFFFFFFFFu, best_c, o);
      if (ob > best_obj || (ob == best_obj && cb < best_c)) {
        best_obj = ob;
        best_c = cb;
      }
    }
    if (tid == 0) sh_best_c = best_c == INT_MAX ? 0 : best_c;
  }
  __syncthreads();
  const int T = p.cand_T[sh_best_c];

  // ---- keep depths: count the selected positions per request ----
  int* counts = reinterpret_cast<int*>(prefix);  // prefix no longer needed
  int* offsets = counts + B;                       // [B]
  for (int i = tid; i < B; i += kAllocThreads) counts[i] = 0;
  __syncthreads();
  for (int q = tid; q < T; q += kAllocThreads) atomicAdd(&counts[0xFFFF - (int)(keys[q] & 0xFFFFull)], 1);
  __syncthreads();

  // ---- row offsets: exclusive scan of (n_i + 1) = counts ----
  const int perB = (B + kAllocThreads - 1) / kAllocThreads;
  const int b0 = tid * perB;
  long long lsum = 0;
  for (int i = b0; i < b0 + perB && i < B; ++i) lsum += counts[i];
  const long long bincl = block_inclusive_scan(lsum, warp_tot);
  long long off = bincl - lsum;
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
      p.packed_tokens_out[row] = k == 0 ? sm.last[i] : sm.drafts[i * K + (k - 1)];
      p.packed_pos_out[row] = sm.pos[i] + k;
    } else {
      p.packed_tokens_out[q] = -1;
      p.packed_pos_out[q] = -1;
    }
  }
  if (tid == 0 && sh_bad) report(p.status, SPEC_ERR_BAD_INPUT);
}

// ---------------------------------------------------------------------------
// Batches of at most 1024 requests and 1024 draft positions (B * K)
// ---------------------------------------------------------------------------
// Every bonus position (k = 0) has the largest score (s = 1) and the smallest
// k, so it ranks above every draft position, and the bonus positions rank
// among themselves by request index.  The global order is therefore the B
// bonus positions, then the B * K draft keys sorted; only the latter need a
// sort.  One draft key per thread, sorted by a bitonic network over 1024 slots
// (padding key 0 ranks below every real key, whose k field is nonzero):
// partners within a warp exchange by shuffles, others through shared memory,
// one barrier per such stage.  The keep depths then follow from the sorted
// ranks without atomics: draft (i, k) in the top T - B, with (i, k + 1) not,
// ends request i's kept prefix.
constexpr int kSmallSlots = kAllocThreads;

// units * 2^-40 as a double, for 0 < units < 2^53 (exact), with integer
// operations only: the product's exponent and mantissa fields are set directly.
__device__ __forceinline__ double units_to_double(long long units) {
  const int msb = 63 - __clzll(units);
  const unsigned long long mant = ((unsigned long long)units << (63 - msb)) << 1 >> 12;  // the bits below the msb
  const unsigned long long expo = (unsigned long long)(msb - 40 + 1023);
  return __longlong_as_double((long long)((expo << 52) | mant));
}

__device__ __forceinline__ unsigned long long shfl_xor_u64(unsigned long long x, int o) {
  const unsigned lo = __shfl_xor_sync(0xFFFFFFFFu, (unsigned)x, o);
  const unsigned hi = __shfl_xor_sync(0xFFFFFFFFu, (unsigned)(x >> 32), o);
  return ((unsigned long long)hi << 32) | lo;
}

// One level of the small kernel's merge tree over kSmallSlots keys in shared
// memory (src), runs of L keys merged in pairs into dst; x is the calling
// thread's key at slot tid, and on return the key at slot tid of the merged
// order (src and dst swapped).
template <int L>
__device__ __forceinline__ void merge_level(unsigned long long& x, int tid, uint32_t& src, uint32_t& dst) {
  const uint32_t partner = src + 8u * (uint32_t)((tid ^ L) & ~(L - 1));
  int c = 0;
#pragma unroll
  for (int step = L >> 1; step > 0; step >>= 1)
    if (lds_u64(partner + 8u * (uint32_t)(c + step - 1)) > x) c += step;
  if (lds_u64(partner + 8u * (uint32_t)c) > x) ++c;
  sts_u64(dst + 8u * (uint32_t)((tid & ~(2 * L - 1)) + (tid & (L - 1)) + c), x);
  __syncthreads();
  const uint32_t t = src;
  src = dst;
  dst = t;
  x = lds_u64(src + 8u * (uint32_t)tid);
}

__global__ void __launch_bounds__(kAllocThreads) allocate_small_kernel(const AllocLaunch p) {
  __shared__ float sh_conf[2 * kSmallSlots];               // [i][k] at i * (K | 1) + k
  __shared__ int32_t sh_drafts[kSmallSlots];
  __shared__ int32_t sh_last[kSmallSlots];
  __shared__ long long sh_pos[kSmallSlots];
  __shared__ unsigned long long sh_x[2][kSmallSlots];      // sort exchanges, then prefix sums / depths
  __shared__ int32_t sh_rank[kSmallSlots];                 // sorted rank of draft (i, k) at i * K + k - 1
  __shared__ long long warp_tot[32];
  __shared__ int sh_best_c, sh_bad;
  const int B = p.B, K = p.K, NK = B * K, CS = K | 1;
  const int tid = threadIdx.x;
  if (tid == 0) sh_bad = 0;
  // The next kernel (the streaming pass) may launch now: it waits for this
  // one's completion before it reads the depths and row offsets.
  pdl_launch_dependents();
  // This kernel starts while the previous one on the stream drains; it reads
  // its inputs, and overwrites the arrays the previous round's kernels read,
  // only once that kernel has completed.
  pdl_wait_prerequisites();

  // ---- every global input in one round trip ----
  if (tid < NK) {
    const int i = tid / K;
    sh_conf[tid + i * (CS - K)] = p.conf[tid];
    sh_drafts[tid] = p.drafts[tid];
  }
  if (tid < B) {
    sh_last[tid] = p.last_tokens[tid];
    sh_pos[tid] = p.pos_base[tid];
  }
  __syncthreads();

  // ---- Eq. (dcut-score): fp32 prefix products, request i in thread i ----
  // When B * KP <= 1024 (KP = the next power of two >= K), request i's keys
  // fill run i of KP slots in descending order (s is non-increasing in k),
  // and the slots past K, and the runs past B, hold pad keys: unique, below
  // every real key, descending within a run.  A merge tree then sorts the
  // 1024 slots.  Otherwise the keys are staged unsorted for a bitonic sort.
  const int KP = K <= 1 ? 1 : 1 << (32 - __clz(K - 1));
  const bool runs = B * KP <= kSmallSlots;
  // Keys are staged with a row of RL slots per request at the odd stride
  // RS = RL + 1 (in 8-byte words), so that the threads of a half-warp, one
  // request each, store to distinct banks.
  const int RL = runs ? KP : (K > 0 ? K : 1), RS = RL + 1;
  unsigned long long* stage = &sh_x[0][0];  // B * RS <= 2048 words over both buffers
  if (tid < B) {
    const float* ci = sh_conf + tid * CS;
    float s = 1.0f;
    for (int k0 = 1; k0 <= K; k0 += 4) {
      float c4[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) c4[u] = k0 + u <= K ? ci[k0 + u - 1] : 1.0f;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int k = k0 + u;
        if (k > K) break;
        float c = c4[u];
        if (!(c >= 0.0f && c <= 1.0f)) {
          sh_bad = 1;
          c = 0.0f;
        }
        c = __fadd_rn(c, 0.0f);  // -0 counts as +0 (its sign bit would break the key order)
        s = __fmul_rn(s, c);
        stage[tid * RS + k - 1] = position_key(s, k, tid);
      }
    }
  }
  __syncthreads();

  unsigned long long x;
  if (runs) {
    // slot u = i * KP + (k - 1); a pad key is 1024 - u (real keys are above
    // 0xFBFF0000 even at s = 0)
    x = (tid / KP < B && tid % KP < K) ? stage[(tid / KP) * RS + tid % KP] : (unsigned long long)(kSmallSlots - tid);
    __syncthreads();  // the staging area holds the merge buffers from here on
    // ---- merge tree, descending: at the level of runs of L keys, a key's
    // place in the merged pair is its index in its run plus the number of
    // keys of the partner run above it (keys are unique), found by a
    // branch-free binary search of log2(L) + 1 shared-memory probes ----
    uint32_t src = (uint32_t)__cvta_generic_to_shared(&sh_x[0][0]);
    uint32_t dst = (uint32_t)__cvta_generic_to_shared(&sh_x[1][0]);
    sts_u64(src + 8u * (uint32_t)tid, x);
    __syncthreads();
    // the levels from runs of KP on, each unrolled for its L
    switch (31 - __clz(KP)) {
      case 0: merge_level<1>(x, tid, src, dst); [[fallthrough]];
      case 1: merge_level<2>(x, tid, src, dst); [[fallthrough]];
      case 2: merge_level<4>(x, tid, src, dst); [[fallthrough]];
      case 3: merge_level<8>(x, tid, src, dst); [[fallthrough]];
      case 4: merge_level<16>(x, tid, src, dst); [[fallthrough]];
      case 5: merge_level<32>(x, tid, src, dst); [[fallthrough]];
      case 6: merge_level<64>(x, tid, src, dst); [[fallthrough]];
      case 7: merge_level<128>(x, tid, src, dst); [[fallthrough]];
      case 8: merge_level<256>(x, tid, src, dst); [[fallthrough]];
      case 9: merge_level<512>(x, tid, src, dst); [[fallthrough]];
      default: break;
    }
  } else {
    // ---- bitonic sort of the draft keys, descending ----
    x = tid < NK ? stage[(tid / RL) * RS + tid % RL] : 0ull;
    __syncthreads();  // the staging area is the exchange buffer from here on
    int buf = 1;
#pragma unroll
    for (int k = 2; k <= kSmallSlots; k <<= 1) {
#pragma unroll
      for (int j = k >> 1; j > 0; j >>= 1) {
        unsigned long long y;
        if (j >= 32) {
          sh_x[buf][tid] = x;
          __syncthreads();
          y = sh_x[buf][tid ^ j];
          buf ^= 1;
        } else {
          y = shfl_xor_u64(x, j);
        }
        // blocks of k alternate direction (descending first); the lower
        // index of a pair keeps the larger key in a descending block
        const bool take_max = ((tid & k) == 0) == ((tid & j) == 0);
        x = take_max ? (x > y ? x : y) : (x < y ? x : y);
      }
    }
  }
  // x: the draft key of rank tid (tid < NK)
  const int xi = 0xFFFF - (int)(x & 0xFFFFull);
  const int xk = 0xFFFF - (int)((x >> 16) & 0xFFFFull);
  if (tid < NK) sh_rank[xi * K + (xk - 1)] = tid;

  // ---- inclusive scan of floor(s * 2^40) over the sorted draft keys ----
  const long long q40 = tid < NK ? (long long)__float2ll_rd(__uint_as_float((unsigned)(x >> 32)) * 0x1p40f) : 0;
  const long long incl = block_inclusive_scan(q40, warp_tot);  // its barriers also end the sort's reads
  long long* prefix = reinterpret_cast<long long*>(sh_x[0]);
  prefix[tid] = incl;
  __syncthreads();

  // ---- Eq. (dcut-select): first maximiser of U / cost ----
  if (tid < 32) {
    long long best_key = -1;
    int best_c = INT_MAX;
    for (int c = tid; c < p.M; c += 32) {
      const int td = p.cand_T[c] - B;  // draft positions kept at this budget
      const long long Uq = ((long long)B << 40) + (td > 0 ? prefix[td - 1] : 0);
      const double U = units_to_double(Uq);
      if (p.utility_out) p.utility_out[c] = U;
      // U > 0 and cost > 0: the bit patterns of the quotients order as the
      // quotients do, so the comparisons below are integer ones
      const long long obj = __double_as_longlong(U / p.cand_cost[c]);
      if (obj > best_key) {  // c increases along the lane's loop
        best_key = obj;
        best_c = c;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const long long ob = __shfl_xor_sync(0xFFFFFFFFu, best_key, o);
      const int cb = __shfl_xor_sync(0xFFFFFFFFu, best_c, o);
      if (ob > best_key || (ob == best_key && cb < best_c)) {
        best_key = ob;
        best_c = cb;
      }
    }
    if (tid == 0) sh_best_c = best_c == INT_MAX ? 0 : best_c;
  }
  int* depth = reinterpret_cast<int*>(sh_x[1]);
  int* offsets = depth + kSmallSlots;
  if (tid < B) depth[tid] = 0;
  __syncthreads();
  const int T = p.cand_T[sh_best_c];
  const int TD = T - B;

  // ---- keep depths: the last kept draft of each request ----
  if (tid < NK && tid < TD) {
    const bool next_kept = xk < K && sh_rank[xi * K + xk] < TD;
    if (!next_kept) depth[xi] = xk;
  }
  __syncthreads();

  // ---- row offsets: exclusive scan of (n_i + 1), one warp: lane l takes
  // the requests [l * m, (l + 1) * m) in order, m = ceil(B / 32) ----
  if (tid < 32) {
    const int m = (B + 31) >> 5;
    const int i0 = min(B, tid * m), i1 = min(B, i0 + m);
    int sum = 0;
    for (int i = i0; i < i1; ++i) sum += depth[i] + 1;
    int incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (tid >= o) incl += y;
    }
    int off = incl - sum;
    for (int i = i0; i < i1; ++i) {
      const int n = depth[i];
      offsets[i] = off;
      p.row_offsets_out[i] = off;
      p.depth_out[i] = n;
      off += n + 1;
    }
    if (tid == 0) {
      p.row_offsets_out[B] = T;  // sum of (n_i + 1): the T kept positions
      *p.chosen_T_out = T;
    }
  }
  __syncthreads();

  // ---- dense packing of the kept prefixes ----
  if (tid < B) {
    p.packed_tokens_out[offsets[tid]] = sh_last[tid];
    p.packed_pos_out[offsets[tid]] = sh_pos[tid];
  }
  if (tid < NK && tid < TD) {
    const int row = offsets[xi] + xk;
    p.packed_tokens_out[row] = sh_drafts[xi * K + (xk - 1)];
    p.packed_pos_out[row] = sh_pos[xi] + xk;
  }
  for (int r = T + tid; r < B * (K + 1); r += kAllocThreads) {
    p.packed_tokens_out[r] = -1;
    p.packed_pos_out[r] = -1;
  }
  if (tid == 0 && sh_bad) report(p.status, SPEC_ERR_BAD_INPUT);
}

bool allocate_is_small(int B, int K) { return B <= kSmallSlots && (long long)B * K <= kSmallSlots; }

cudaError_t launch_allocate(const AllocLaunch& p, cudaStream_t stream) {
  cudaError_t err;
  if (allocate_is_small(p.B, p.K)) {
    err = launch_after_previous(allocate_small_kernel, dim3(1), dim3(kAllocThreads), 0, stream, p);
    return err != cudaSuccess ? err : cudaGetLastError();
  }
  // The dynamic shared memory limit is raised once per device, to the
  // largest size asked for so far.
  const size_t smem = allocate_smem_bytes(p.B, p.K);
  constexpr int kMaxDevices = 64;
  static std::atomic<size_t> raised[kMaxDevices];
  int dev = -1;
  err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (dev < 0 || dev >= kMaxDevices || raised[dev].load(std::memory_order_relaxed) < smem) {
    err = cudaFuncSetAttribute(allocate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    if (dev >= 0 && dev < kMaxDevices) {
      size_t cur = raised[dev].load(std::memory_order_relaxed);
      while (cur < smem && !raised[dev].compare_exchange_weak(cur, smem)) {
      }
    }
  }
  err = launch_after_previous(allocate_kernel, dim3(1), dim3(kAllocThreads), smem, stream, p);
  return err != cudaSuccess ? err : cudaGetLastError();
}

}  // namespace spec
