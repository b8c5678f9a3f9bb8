// draft.cu -- the drafter's producer step on sm_103a: drafts, token-level
// confidences and D-cut scores from the drafter's logits in one streaming
// pass (arxiv 2607.25852, Section 4.2: D-cut ranks positions by the prefix
// products s_{i,k} of the drafter's confidences c_{i,t}, Eq. dcut-score).
//
// Row k of request i holds the drafter's logits for draft z_{k+1}:
//   q_k = softmax(l_k / tau)                     (tau' = tau, or 1 at tau = 0)
//   z_{k+1} ~ q_k by the two-level exponential race at position
//             pos_base_i + k + 1, purposes DRAFT / DRAFT_IN_BLOCK
//             (argmax, lowest index, at tau = 0)
//   c_{k+1} = q_k(z_{k+1}) at tau'
//   s_0 = 1, s_k = fl32(s_{k-1} * c_k)
//
// draft_rows_kernel: one CTA per (row, chunk of equal size).  Each
// warp takes a round of 8 consecutive race blocks (256 entries each; 4 for
// fp32) at a time: lane l loads entries 8l..8l+7 of each, the round's max
// comes from one redux over order-preserving integer keys, and the blocks'
// sums of 2^(l*c2 - fl(M_r*c2)) from one transposed butterfly, after which
// each group of lanes owns one block.  Level 1 of the race compares blocks in
// the log2 domain,
//   log2 key_b = log2 E_b - log2 sum_b - M_r*c2   (see BlockKey),
// so no pass over the row is needed before the draw.  The row's softmax
// statistics merge from the rounds' (M_r, sum_r).  The last CTA of a row to
// arrive merges the chunks, draws the entry inside the winning block (level
// 2) and writes z, c and the row statistics; the last row of a request to
// finish writes the scores.
#include <float.h>
#include <math.h>

#include <algorithm>

#include "verify_common.cuh"

namespace spec {

constexpr int kDraftThreads = 256;
constexpr int kSegmentBlocks = 64;  // race blocks per warp unit, at most

// A level-1 candidate: block idx with L = log2 E_b - log2 sum_b and block
// max M, i.e. log2 key = L - M*c2.  Two candidates compare by
// L_a - L_b < c2 * (M_a - M_b): the rounding then scales with the gap between
// the two maxima, not with |M*c2| (which reaches hundreds at small tau).
struct BlockKey {
  float L, M;
  int32_t idx;  // INT_MAX: none
};
__device__ __forceinline__ bool block_key_better(const BlockKey& a, const BlockKey& b, float c2) {
  if (a.idx == INT_MAX) return false;
  if (b.idx == INT_MAX) return true;
  const float lhs = a.L - b.L, rhs = c2 * (a.M - b.M);
  return lhs < rhs || (lhs == rhs && a.idx < b.idx);
}

struct alignas(16) DraftPartial {
  float m;        // max logit of the chunk
  float s;        // sum of 2^(l*c2 - fl(m*c2))
  float key;      // tau > 0: L of the best block; tau = 0: the max (= m)
  int32_t idx;    // tau > 0: the best block; tau = 0: lowest argmax (INT_MAX: none)
  int32_t flags;  // bit0: NaN or +inf seen
  float keyM;     // tau > 0: M of the best block
  int32_t pad[2];
};

struct DraftLaunch {
  const void* logits;  // [B*K, V]
  int B, K, V;
  float tau, c2, inv_t;  // c2 = log2(e) / tau'
  const uint64_t* seeds;
  const uint64_t* request_ids;
  const int64_t* pos_base;
  int32_t* drafts;     // [B, K]
  float* conf;         // [B, K]
  float* scores;       // [B, K+1] or null
  float* row_stats;    // [B*K, 2] or null
  int32_t* status;
  DraftPartial* part;  // [B*K*NC]
  uint32_t* row_count; // [B*K]
  uint32_t* req_count; // [B]
  uint32_t* req_bad;   // [B]
  int NC, chunk;       // segments per row (one warp each), entries per segment (a multiple of 2048)
};

struct DraftGeometry {
  int NC, chunk;
  size_t part_off, counters_off, bytes;
};

static inline long long ceil_div_ll(long long a, long long b) { return (a + b - 1) / b; }

static DraftGeometry draft_geometry(int B, int K, int V) {
  DraftGeometry g{};
  const long long R = (long long)B * K;
  // one warp per (row, segment): segments of about 64 blocks (8 rounds),
  // split evenly in steps of 8 blocks
  const long long nb = ceil_div_ll(V, 256);
  const long long ns = std::max(1LL, ceil_div_ll(nb, kSegmentBlocks));
  const long long bps = std::min<long long>(kSegmentBlocks, ceil_div_ll(ceil_div_ll(nb, ns), 8) * 8);
  g.NC = (int)ceil_div_ll(nb, bps);
  g.chunk = (int)(bps * 256);
  g.part_off = 0;
  g.counters_off = ((size_t)sizeof(DraftPartial) * R * g.NC + 255) / 256 * 256;
  g.bytes = g.counters_off + ((size_t)sizeof(uint32_t) * (R + 2 * (size_t)B) + 255) / 256 * 256;
  return g;
}

__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Order-preserving map of a non-NaN float onto int32 (signed compare).
__device__ __forceinline__ int orderable(float f) {
  const int b = __float_as_int(f);
  return b < 0 ? b ^ 0x7FFFFFFF : b;
}
__device__ __forceinline__ float from_orderable(int k) { return __int_as_float(k < 0 ? k ^ 0x7FFFFFFF : k); }

// A lane's 8 entries 8l..8l+7 of a race block as raw 16-byte words (one for
// bf16, two for fp32), and their unpacking; entries at or past V read -inf.
template <typename T>
struct Lane8;
template <>
struct Lane8<__nv_bfloat16> {
  static constexpr int kWords = 1;
  static constexpr int kBlocksPerRound = 8;  // two Philox quads
  template <bool kVec>
  __device__ static void load(const __nv_bfloat16* row, int v8, int V, uint4 (&w)[kWords]) {
    if (kVec) {
      w[0] = v8 < V ? ldg_stream(row + v8) : make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
    } else {
      uint32_t h[8];
#pragma unroll
      for (int e = 0; e < 8; ++e)
        h[e] = v8 + e < V ? (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(row) + v8 + e) : 0xFF80u;
      w[0] = make_uint4(h[0] | h[1] << 16, h[2] | h[3] << 16, h[4] | h[5] << 16, h[6] | h[7] << 16);
    }
  }
  __device__ static void unpack(const uint4 (&w)[kWords], float (&x)[8]) {
    x[0] = bf16_lo(w[0].x), x[1] = bf16_hi(w[0].x), x[2] = bf16_lo(w[0].y), x[3] = bf16_hi(w[0].y);
    x[4] = bf16_lo(w[0].z), x[5] = bf16_hi(w[0].z), x[6] = bf16_lo(w[0].w), x[7] = bf16_hi(w[0].w);
  }
  // max over the lane's entries of N blocks as a tree of packed bf16 maxima
  // (a NaN loses to any number here; the sums catch it)
  template <int N>
  __device__ static float round_max(const uint4 (&w)[N][kWords]) {
    __nv_bfloat162 m[N];
#pragma unroll
    for (int u = 0; u < N; ++u) {
      const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&w[u][0]);
      m[u] = __hmax2(__hmax2(h[0], h[1]), __hmax2(h[2], h[3]));
    }
#pragma unroll
    for (int n = N / 2; n > 0; n >>= 1)
#pragma unroll
      for (int u = 0; u < n; ++u) m[u] = __hmax2(m[u], m[u + n]);
    return fmaxf(__low2float(m[0]), __high2float(m[0]));
  }
};
template <>
struct Lane8<float> {
  static constexpr int kWords = 2;
  static constexpr int kBlocksPerRound = 4;  // one Philox quad
  template <bool kVec>
  __device__ static void load(const float* row, int v8, int V, uint4 (&w)[kWords]) {
    const uint32_t ninf = 0xFF800000u;
    if (kVec) {
      w[0] = v8 < V ? ldg_stream(row + v8) : make_uint4(ninf, ninf, ninf, ninf);
      w[1] = v8 < V ? ldg_stream(row + v8 + 4) : make_uint4(ninf, ninf, ninf, ninf);
    } else {
      uint32_t h[8];
#pragma unroll
      for (int e = 0; e < 8; ++e)
        h[e] = v8 + e < V ? __float_as_uint(__ldg(row + v8 + e)) : ninf;
      w[0] = make_uint4(h[0], h[1], h[2], h[3]);
      w[1] = make_uint4(h[4], h[5], h[6], h[7]);
    }
  }
  __device__ static void unpack(const uint4 (&w)[kWords], float (&x)[8]) {
    x[0] = __uint_as_float(w[0].x), x[1] = __uint_as_float(w[0].y), x[2] = __uint_as_float(w[0].z);
    x[3] = __uint_as_float(w[0].w), x[4] = __uint_as_float(w[1].x), x[5] = __uint_as_float(w[1].y);
    x[6] = __uint_as_float(w[1].z), x[7] = __uint_as_float(w[1].w);
  }
  template <int N>
  __device__ static float round_max(const uint4 (&w)[N][kWords]) {
    float m[N];
#pragma unroll
    for (int u = 0; u < N; ++u) {
      float x[8];
      unpack(w[u], x);
      m[u] = fmaxf(fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3])), fmaxf(fmaxf(x[4], x[5]), fmaxf(x[6], x[7])));
    }
#pragma unroll
    for (int n = N / 2; n > 0; n >>= 1)
#pragma unroll
      for (int u = 0; u < n; ++u) m[u] = fmaxf(m[u], m[u + n]);
    return m[0];
  }
};

// Per-warp state of a chunk (identical in every lane).
struct WarpDraftState {
  SoftState st{-INFINITY, 0.0f};
  BlockKey best{INFINITY, 0.0f, INT_MAX};  // tau > 0
  ArgState g{-INFINITY, INT_MAX};          // tau = 0: (max, lowest index)
  int32_t flags = 0;
};

// Sum of per-lane values acc[u] (u < N, N = 4 or 8: one per race block of
// the round) over the warp, transposed: after log2 N halving exchanges and a
// butterfly over the remaining lane bits, lane l holds the sum of block
// l >> (5 - log2 N); the 32 / N lanes of a block hold identical values.
template <int N>
__device__ __forceinline__ float transposed_block_sum(const float (&acc)[N], int lane) {
  static_assert(N == 4 || N == 8, "4 or 8 blocks per round");
  float v[N];
#pragma unroll
  for (int u = 0; u < N; ++u) v[u] = acc[u];
#pragma unroll
  for (int n = N, o = 16; n > 1; n >>= 1, o >>= 1) {
    const bool hi = (lane & o) != 0;
#pragma unroll
    for (int j = 0; j < n / 2; ++j) {
      const float send = hi ? v[j] : v[j + n / 2];
      const float keep = hi ? v[j + n / 2] : v[j];
      v[j] = keep + __shfl_xor_sync(0xFFFFFFFFu, send, o);
    }
  }
#pragma unroll
  for (int o = 16 / N; o > 0; o >>= 1) v[0] += __shfl_xor_sync(0xFFFFFFFFu, v[0], o);
  return v[0];
}

// soft_merge with the scale factor from ex2.approx (relative error ~2^-22):
// the per-round merges of the streaming softmax.
__device__ __forceinline__ SoftState soft_merge_fast(SoftState a, SoftState b, float c2) {
  if (b.m > a.m) {
    const SoftState t = a;
    a = b;
    b = t;
  }
  if (b.m == -INFINITY) return a;
  a.s = a.s + b.s * ex2_approx(b.m * c2 - a.m * c2);
  return a;
}

// The level-1 race words of blocks g0 .. g0+31 (g0 a multiple of 32), lane
// l holding block g0 + l's: word l & 3 of the Philox quad at counter
// (g0 >> 2) + (l >> 2).  One quad per lane serves 32 / N rounds.
__device__ __forceinline__ uint32_t race_words(int g0, int lane, uint32_t position, uint64_t req, uint32_t k0,
                                               uint32_t k1) {
  const uint4 rq = philox(draw_counter(position, req, SPEC_PURPOSE_DRAFT, (uint32_t)((g0 >> 2) + (lane >> 2))), k0, k1);
  const int e = lane & 3;
  return e == 0 ? rq.x : e == 1 ? rq.y : e == 2 ? rq.z : rq.w;
}

// One round of N consecutive race blocks b0 .. b0+N-1 of the warp (blocks at
// or past b_hi were loaded as -inf).  Every value is taken relative to the
// round's max M_r: the blocks' sums of 2^(l*c2 - fl(M_r*c2)) (a block whose
// weight underflows against M_r is more than 2^-126 below the round's best
// and cannot win the race), the round's softmax contribution, and each
// block's level-1 candidate (L = log2 E_b - log2 sum_b, M = M_r), one block
// per lane group.  Lane l's `rword` is the race word of block g0 + l, g0 the
// first block of the group of 32 that holds this round (race_words).
template <typename T, bool kGreedy>
__device__ __forceinline__ void draft_round(WarpDraftState& ws, const uint4 (&w)[Lane8<T>::kBlocksPerRound][Lane8<T>::kWords],
                                            int b0, int b_hi, int lane, float c2, uint32_t rword) {
  using L8 = Lane8<T>;
  constexpr int N = L8::kBlocksPerRound;
  // ---- the round's max (+inf makes the row unusable; a NaN is caught by
  // the sums below, which it turns into NaN) ----
  const float lmax = L8::template round_max<N>(w);
  const float Mr = from_orderable(__reduce_max_sync(0xFFFFFFFFu, orderable(lmax)));
  if (Mr == INFINITY) {
    ws.flags |= 1;
    return;
  }
  if (Mr == -INFINITY) {  // no finite entry in the round: weight 0, unless a NaN hides here
    bool nan = false;
#pragma unroll
    for (int u = 0; u < N; ++u) {
      float x[8];
      L8::unpack(w[u], x);
#pragma unroll
      for (int e = 0; e < 8; ++e) nan |= x[e] != x[e];
    }
    if (__any_sync(0xFFFFFFFFu, nan)) ws.flags |= 1;
    return;
  }
  if (kGreedy && (ws.g.idx == INT_MAX || Mr > ws.g.v)) {
    // a new running max: its first index (rounds arrive in increasing order)
    unsigned first = 0xFFFFFFFFu;
#pragma unroll
    for (int u = N - 1; u >= 0; --u) {
      float x[8];
      L8::unpack(w[u], x);
#pragma unroll
      for (int e = 7; e >= 0; --e)
        if (x[e] == Mr) first = (unsigned)((b0 + u) * kRaceBlock + 8 * lane + e);
    }
    ws.g = ArgState{Mr, (int)__reduce_min_sync(0xFFFFFFFFu, first)};
  }
  // ---- per-block sums relative to the round's max ----
  const float M2 = Mr * c2;
  const float2 c2v = make_float2(c2, c2), nM2 = make_float2(-M2, -M2);
  float acc[N];
#pragma unroll
  for (int u = 0; u < N; ++u) {
    float x[8];
    L8::unpack(w[u], x);
    float2 a0 = make_float2(0.f, 0.f), a1 = make_float2(0.f, 0.f);
#pragma unroll
    for (int e = 0; e < 8; e += 4) {
      const float2 y0 = __ffma2_rn(make_float2(x[e], x[e + 1]), c2v, nM2);
      const float2 y1 = __ffma2_rn(make_float2(x[e + 2], x[e + 3]), c2v, nM2);
      a0 = __fadd2_rn(a0, make_float2(ex2_approx(y0.x), ex2_approx(y0.y)));
      a1 = __fadd2_rn(a1, make_float2(ex2_approx(y1.x), ex2_approx(y1.y)));
    }
    acc[u] = (a0.x + a0.y) + (a1.x + a1.y);
  }
  const int ub = lane >> (N == 8 ? 2 : 3);  // this lane's block of the round
  const float sb = transposed_block_sum<N>(acc, lane);
  float sr = sb;  // the round's sum: add the N distinct blocks
#pragma unroll
  for (int o = 32 / N; o < 32; o <<= 1) sr += __shfl_xor_sync(0xFFFFFFFFu, sr, o);
  if (sr != sr) {  // a NaN entry
    ws.flags |= 1;
    return;
  }
  ws.st = soft_merge_fast(ws.st, SoftState{Mr, sr}, c2);
  if (kGreedy) return;
  // ---- level-1 candidates, one block per lane group ----
  const int b = b0 + ub;
  const uint32_t word = __shfl_sync(0xFFFFFFFFu, rword, b & 31);
  // E near 0 needs log1pf; log2 of E and of the sum go to lg2.approx, whose
  // absolute error (~1e-7) is what a log-domain key can afford
  KeyState cand{INFINITY, INT_MAX};
  if (b < b_hi && sb > 0.0f) {
    const float E = -log1pf(-((float)race_m(word) * 0x1p-24f));
    cand = KeyState{lg2_approx(E) - lg2_approx(sb), b};
  }
  // every candidate of the round shares M = M_r: compare L alone
#pragma unroll
  for (int o = 32 / N; o < 32; o <<= 1) {
    const KeyState other{__shfl_xor_sync(0xFFFFFFFFu, cand.key, o), __shfl_xor_sync(0xFFFFFFFFu, cand.idx, o)};
    if (key_better(other, cand)) cand = other;
  }
  if (cand.idx != INT_MAX) {
    const BlockKey rb{cand.key, Mr, cand.idx};
    if (block_key_better(rb, ws.best, c2)) ws.best = rb;
  }
}

// Minimum key over the warp (every lane).
__device__ __forceinline__ KeyState warp_min_key(KeyState b) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const KeyState other{__shfl_xor_sync(0xFFFFFFFFu, b.key, o), __shfl_xor_sync(0xFFFFFFFFu, b.idx, o)};
    if (key_better(other, b)) b = other;
  }
  return b;
}

// One warp per (row, segment of SB blocks); the warps of a CTA are
// independent (no CTA barrier).  The last warp of a row to arrive merges the
// row's segment partials, draws inside the winning block and writes the
// row's outputs; the last row of a request writes the scores.
template <typename T, bool kGreedy, bool kVec>
__global__ void __launch_bounds__(kDraftThreads, 4) draft_rows_kernel(const DraftLaunch p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long unit = (long long)blockIdx.x * (kDraftThreads / 32) + warp;
  pdl_wait_prerequisites();
  pdl_launch_dependents();
  if (unit >= (long long)p.B * p.K * p.NC) return;
  const int r = (int)(unit / p.NC);
  const int c = (int)(unit - (long long)r * p.NC);
  const int i = r / p.K;
  const int k = r - i * p.K;
  const T* row = static_cast<const T*>(p.logits) + (size_t)r * (size_t)p.V;

  // ---- this segment's blocks, a round of consecutive ones at a time ----
  const int nb = (p.V + kRaceBlock - 1) / kRaceBlock;
  const int bps = p.chunk / kRaceBlock;
  const int b_lo = c * bps, b_hi = min(nb, b_lo + bps);
  using L8 = Lane8<T>;
  constexpr int kBPR = L8::kBlocksPerRound;
  uint4 w[kBPR][L8::kWords];
  auto load_round = [&](int b0) {
#pragma unroll
    for (int u = 0; u < kBPR; ++u)
      L8::template load<kVec>(row, (b0 + u) * kRaceBlock + 8 * lane, b0 + u < b_hi ? p.V : 0, w[u]);
  };
  if (b_lo < b_hi) load_round(b_lo);  // the first loads ahead of the request's scalars
  const long long pos = __ldg(reinterpret_cast<const long long*>(p.pos_base) + i);
  const bool pos_ok = pos >= 0 && pos + p.K <= 0xFFFFFFFFLL;
  const uint32_t position = (uint32_t)(pos + k + 1);
  const uint64_t req = __ldg(reinterpret_cast<const unsigned long long*>(p.request_ids) + i);
  const uint64_t seed = __ldg(reinterpret_cast<const unsigned long long*>(p.seeds) + i);
  const uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
  WarpDraftState ws;
  uint32_t rword = 0;
  for (int b0 = b_lo; b0 < b_hi; b0 += kBPR) {
    if (b0 != b_lo) load_round(b0);
    if (!kGreedy && (b0 == b_lo || (b0 & 31) == 0)) rword = race_words(b0 & ~31, lane, position, req, k0, k1);
    draft_round<T, kGreedy>(ws, w, b0, b_hi, lane, p.c2, rword);
  }

  // ---- the segment's partial; the last warp of the row goes on ----
  int last = 0;
  if (lane == 0) {
    DraftPartial d{};
    d.m = ws.st.m;
    d.s = ws.st.s;
    d.key = kGreedy ? ws.g.v : ws.best.L;
    d.keyM = kGreedy ? 0.0f : ws.best.M;
    d.idx = kGreedy ? ws.g.idx : ws.best.idx;
    d.flags = ws.flags;
    p.part[(size_t)r * p.NC + c] = d;
    __threadfence();  // the partial before the count
    last = atomicAdd(p.row_count + r, 1u) == (uint32_t)(p.NC - 1);
  }
  if (!__shfl_sync(0xFFFFFFFFu, last, 0)) return;
  __threadfence();  // the other segments' partials after their counts

  // ---- merge the row's segments (lanes over segments) ----
  SoftState st{-INFINITY, 0.0f};
  BlockKey best{INFINITY, 0.0f, INT_MAX};
  ArgState g{-INFINITY, INT_MAX};
  int32_t f = 0;
  for (int cc = lane; cc < p.NC; cc += 32) {
    const uint4* src = reinterpret_cast<const uint4*>(p.part + (size_t)r * p.NC + cc);
    const uint4 a = __ldcg(src), b2 = __ldcg(src + 1);
    st = soft_merge(st, SoftState{__uint_as_float(a.x), __uint_as_float(a.y)}, p.c2);
    if (kGreedy) {
      const ArgState o{__uint_as_float(a.z), (int32_t)a.w};
      if (arg_better(o, g)) g = o;
    } else {
      const BlockKey o{__uint_as_float(a.z), __uint_as_float(b2.y), (int32_t)a.w};
      if (block_key_better(o, best, p.c2)) best = o;
    }
    f |= (int32_t)b2.x;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    st = soft_merge(st, SoftState{__shfl_xor_sync(0xFFFFFFFFu, st.m, o), __shfl_xor_sync(0xFFFFFFFFu, st.s, o)},
                    p.c2);
    const BlockKey ob{__shfl_xor_sync(0xFFFFFFFFu, best.L, o), __shfl_xor_sync(0xFFFFFFFFu, best.M, o),
                      __shfl_xor_sync(0xFFFFFFFFu, best.idx, o)};
    if (block_key_better(ob, best, p.c2)) best = ob;
    const ArgState og{__shfl_xor_sync(0xFFFFFFFFu, g.v, o), __shfl_xor_sync(0xFFFFFFFFu, g.idx, o)};
    if (arg_better(og, g)) g = og;
  }
  f = (int32_t)__reduce_or_sync(0xFFFFFFFFu, (unsigned)f);
  if (lane == 0) p.row_count[r] = 0u;  // leave the workspace zeroed for the next call
  const int idx = kGreedy ? g.idx : best.idx;
  const bool bad = f || !pos_ok || !(st.m > -INFINITY) || !(st.s > 0.0f) || !isfinite(st.s) || idx == INT_MAX;
  const float M2 = st.m * p.c2;
  int z = -1;
  if (!bad) {
    if (kGreedy) {
      z = idx;
    } else {
      // level 2 in the winning block (8 entries per lane), weights relative
      // to the row max
      KeyState e{INFINITY, INT_MAX};
      const int v0 = idx * kRaceBlock + 8 * lane;
      uint4 rw[2];
      rw[0] = philox(draw_counter(position, req, SPEC_PURPOSE_DRAFT_IN_BLOCK, (uint32_t)(v0 >> 2)), k0, k1);
      rw[1] = philox(draw_counter(position, req, SPEC_PURPOSE_DRAFT_IN_BLOCK, (uint32_t)(v0 >> 2) + 1u), k0, k1);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int v = v0 + j;
        if (v < p.V) {
          const float wv = ex2_approx(__fmaf_rn(load_elem(row + v), p.c2, -M2));
          const uint4& q4 = rw[j >> 2];
          const uint32_t word = (j & 3) == 0 ? q4.x : (j & 3) == 1 ? q4.y : (j & 3) == 2 ? q4.z : q4.w;
          if (wv > 0.0f) {
            const KeyState kv{race_key(race_m(word), wv), v};
            if (key_better(kv, e)) e = kv;
          }
        }
      }
      e = warp_min_key(e);
      z = e.idx == INT_MAX ? -1 : e.idx;
    }
  }
  if (lane != 0) return;
  const size_t o = (size_t)i * p.K + k;
  if (bad || z < 0) {
    p.drafts[o] = -1;
    p.conf[o] = 0.0f;
    if (p.row_stats) reinterpret_cast<float2*>(p.row_stats)[o] = make_float2(0.0f, 0.0f);
    atomicOr(p.req_bad + i, 1u);
  } else {
    p.drafts[o] = z;
    // c = q(z) = 2^(l_z*c2 - fl(m*c2)) / S, with one rounding in the exponent
    p.conf[o] = exp2f(fmaf(load_elem(row + z), p.c2, -M2)) / st.s;
    if (p.row_stats) {
      const float resid = fmaf(st.m, p.c2, -M2);
      reinterpret_cast<float2*>(p.row_stats)[o] = make_float2(st.m * p.inv_t, (log2f(st.s) - resid) * 0.69314718055994531f);
    }
  }
  // ---- the last row of the request: the scores ----
  __threadfence();  // this row's outputs before the count
  if (atomicAdd(p.req_count + i, 1u) != (uint32_t)(p.K - 1)) return;
  __threadfence();
  p.req_count[i] = 0u;
  const bool req_bad = __ldcg(p.req_bad + i) != 0u;
  if (req_bad) {
    p.req_bad[i] = 0u;
    report(p.status, SPEC_ERR_BAD_INPUT);
    for (int kk = 0; kk < p.K; ++kk) {
      p.drafts[(size_t)i * p.K + kk] = -1;
      p.conf[(size_t)i * p.K + kk] = 0.0f;
      if (p.row_stats) reinterpret_cast<float2*>(p.row_stats)[(size_t)i * p.K + kk] = make_float2(0.0f, 0.0f);
    }
  }
  if (p.scores) {
    float* sc = p.scores + (size_t)i * (p.K + 1);
    float run = 1.0f;
    sc[0] = run;
    for (int kk = 0; kk < p.K; ++kk) {
      run = req_bad ? 0.0f : __fmul_rn(run, __ldcg(p.conf + (size_t)i * p.K + kk));
      sc[kk + 1] = run;
    }
  }
}

template <typename T>
static cudaError_t launch_draft_typed(const DraftLaunch& p, bool vec, cudaStream_t stream) {
  const long long units = (long long)p.B * p.K * p.NC;  // one warp each
  const dim3 grid((unsigned)((units + kDraftThreads / 32 - 1) / (kDraftThreads / 32))), block(kDraftThreads);
  const bool greedy = p.tau == 0.0f;
  if (vec)
    return greedy ? launch_after_previous(draft_rows_kernel<T, true, true>, grid, block, 0, stream, p)
                  : launch_after_previous(draft_rows_kernel<T, false, true>, grid, block, 0, stream, p);
  return greedy ? launch_after_previous(draft_rows_kernel<T, true, false>, grid, block, 0, stream, p)
                : launch_after_previous(draft_rows_kernel<T, false, false>, grid, block, 0, stream, p);
}

}  // namespace spec

extern "C" size_t spec_draft_workspace(int B, int K, int V) {
  if (B < 1 || K < 1 || K > SPEC_MAX_DRAFTS || V < 1 || V >= SPEC_MAX_VOCAB || (long long)B * K > (1LL << 28))
    return 0;
  return spec::draft_geometry(B, K, V).bytes;
}

extern "C" int spec_draft(const void* logits, int logits_dtype, int B, int K, int V, float tau,
                          const uint64_t* seeds, const uint64_t* request_ids, const int64_t* pos_base,
                          int32_t* drafts_out, float* conf_out, float* scores_out, float* row_stats_out,
                          int32_t* status, void* ws, size_t ws_bytes, cudaStream_t stream) {
  spec::NvtxRange range("spec_draft");
  if (B < 1 || K < 1 || K > SPEC_MAX_DRAFTS || V < 1 || V >= SPEC_MAX_VOCAB || (long long)B * K > (1LL << 28))
    return SPEC_ERR_INVALID_ARG;
  if ((logits_dtype != SPEC_BF16 && logits_dtype != SPEC_F32) || !(tau >= 0.0f) || isinf(tau))
    return SPEC_ERR_INVALID_ARG;
  if (!logits || !seeds || !request_ids || !pos_base || !drafts_out || !conf_out) return SPEC_ERR_INVALID_ARG;
  if (row_stats_out && (reinterpret_cast<uintptr_t>(row_stats_out) & 7u) != 0) return SPEC_ERR_INVALID_ARG;
  const spec::DraftGeometry g = spec::draft_geometry(B, K, V);
  if (!ws || ws_bytes < g.bytes || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return SPEC_ERR_WORKSPACE;
  spec::DraftLaunch p{};
  p.logits = logits;
  p.B = B;
  p.K = K;
  p.V = V;
  p.tau = tau;
  const double tc = tau > 0.0f ? (double)tau : 1.0;
  p.c2 = (float)(1.4426950408889634 / tc);
  p.inv_t = (float)(1.0 / tc);
  p.seeds = seeds;
  p.request_ids = request_ids;
  p.pos_base = pos_base;
  p.drafts = drafts_out;
  p.conf = conf_out;
  p.scores = scores_out;
  p.row_stats = row_stats_out;
  p.status = status;
  char* base = static_cast<char*>(ws);
  p.part = reinterpret_cast<spec::DraftPartial*>(base + g.part_off);
  const size_t R = (size_t)B * K;
  p.row_count = reinterpret_cast<uint32_t*>(base + g.counters_off);
  p.req_count = p.row_count + R;
  p.req_bad = p.req_count + B;
  p.NC = g.NC;
  p.chunk = g.chunk;
  const size_t esize = logits_dtype == SPEC_F32 ? 4 : 2;
  // 16-byte loads of each lane's 8 entries: aligned rows and whole 8-entry groups
  const bool vec = (reinterpret_cast<uintptr_t>(logits) & 15u) == 0 && ((size_t)V * esize) % 16 == 0 && V % 8 == 0;
  const cudaError_t err = logits_dtype == SPEC_F32 ? spec::launch_draft_typed<float>(p, vec, stream)
                                                   : spec::launch_draft_typed<__nv_bfloat16>(p, vec, stream);
  if (err != cudaSuccess || cudaGetLastError() != cudaSuccess) return SPEC_ERR_CUDA;
  return SPEC_OK;
}
