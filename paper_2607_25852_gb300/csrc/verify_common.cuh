// verify_common.cuh -- device code shared by the verification kernels of
// libspec (verify.cu: the whole-vocabulary path; shard.cu: the
// vocabulary-sharded path): per-thread streaming states and their merges, the
// 16-byte row loaders and the two-level exponential race.  Not part of the
// public ABI.
#pragma once

#include <float.h>
#include <limits.h>
#include <math.h>

#include "spec_internal.cuh"

namespace spec {

constexpr int kStreamThreads = 256;
constexpr int kUnroll = 8;
constexpr int kSampleThreads = 256;
constexpr int kMaxRows = SPEC_MAX_DRAFTS + 1;

// ---------------------------------------------------------------------------
// Per-thread states and their merges
// ---------------------------------------------------------------------------
struct SoftState {
  float m;  // max logit seen
  float s;  // sum of 2^(l*c2 - fl(m*c2))
};

__device__ __forceinline__ SoftState soft_merge(SoftState a, SoftState b, float c2) {
  if (b.m > a.m) {
    SoftState t = a;
    a = b;
    b = t;
  }
  if (b.m == -INFINITY) return a;
  const float Ma = a.m * c2, Mb = b.m * c2;
  a.s = a.s + b.s * exp2f(Mb - Ma);
  return a;
}

struct ArgState {
  float v;
  int32_t idx;  // INT_MAX: nothing seen
};

__device__ __forceinline__ bool arg_better(ArgState a, ArgState b) {
  if (a.idx == INT_MAX) return false;
  if (b.idx == INT_MAX) return true;
  return a.v > b.v || (a.v == b.v && a.idx < b.idx);
}

struct KeyState {
  float key;
  int32_t idx;  // INT_MAX: nothing seen
};

__device__ __forceinline__ bool key_better(KeyState a, KeyState b) {
  return a.key < b.key || (a.key == b.key && a.idx < b.idx);
}

// Barrier over the kThreads threads of a streaming CTA.
template <int kThreads = kStreamThreads>
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kThreads) : "memory");
}

// ---------------------------------------------------------------------------
// Streaming pass
// ---------------------------------------------------------------------------
template <typename T>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int N = 8;
  static constexpr uint32_t kPad = 0xFF80FF80u;  // two bf16 -inf
  __device__ static float get(const uint4& w, int e) {
    const uint32_t word = e < 2 ? w.x : e < 4 ? w.y : e < 6 ? w.z : w.w;
    return (e & 1) ? bf16_hi(word) : bf16_lo(word);
  }
  // NaN-propagating max over the vector (returns NaN if any element is NaN)
  __device__ static float vmax(const uint4& w) {
    __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&w.x);
    a = __hmax2_nan(a, *reinterpret_cast<const __nv_bfloat162*>(&w.y));
    a = __hmax2_nan(a, *reinterpret_cast<const __nv_bfloat162*>(&w.z));
    a = __hmax2_nan(a, *reinterpret_cast<const __nv_bfloat162*>(&w.w));
    return fmax_nan(__low2float(a), __high2float(a));
  }
};
template <>
struct Vec<float> {
  static constexpr int N = 4;
  static constexpr uint32_t kPad = 0xFF800000u;  // fp32 -inf
  __device__ static float get(const uint4& w, int e) {
    const uint32_t word = e == 0 ? w.x : e == 1 ? w.y : e == 2 ? w.z : w.w;
    return __uint_as_float(word);
  }
  __device__ static float vmax(const uint4& w) {
    return fmax_nan(fmax_nan(__uint_as_float(w.x), __uint_as_float(w.y)),
                    fmax_nan(__uint_as_float(w.z), __uint_as_float(w.w)));
  }
};

// Per-thread state of a streamed chunk: softmax (m, s = sum 2^(l*c2 - fl(m*c2)))
// at t > 0, lowest argmax at t = 0; flags bit 0 = NaN (or +inf at t > 0) seen.
// At t = 0 the thread keeps the first 16-byte vector that holds its maximum
// and locates the element inside it once, when the chunk ends (finalize).
template <typename T, bool kGreedy>
struct RowAcc {
  int32_t flags = 0;
  ArgState g{-INFINITY, INT_MAX};
  SoftState st{-INFINITY, 0.0f};
  float M2 = -INFINITY;    // fl(st.m * c2)
  uint4 g_word{0u, 0u, 0u, 0u};  // t = 0: the vector holding the maximum ...
  int g_v0 = INT_MAX;            // ... and the index of its first element

  __device__ __forceinline__ void scalar(int v, float x, float c2) {
    if (x != x) {
      flags |= 1;
      return;
    }
    if (kGreedy) {
      if (g.idx == INT_MAX || x > g.v) {  // a tie keeps the earlier element
        g.v = x;
        g.idx = v;
        g_v0 = INT_MAX;
      }
    } else {
      if (x == INFINITY) flags |= 1;
      if (x > st.m) {
        const float M2n = x * c2;
        st.s = st.s * exp2f(M2 - M2n);
        st.m = x;
        M2 = M2n;
      }
      if (st.m != -INFINITY) st.s += ex2_approx(fmaf(x, c2, -M2));
    }
  }

  // t = 0: resolve the kept vector into (max, lowest index); call once the
  // thread's last element is in.
  __device__ __forceinline__ void finalize() {
    using VT = Vec<T>;
    if (!kGreedy || g_v0 == INT_MAX) return;
    int found = INT_MAX;
#pragma unroll
    for (int e = VT::N - 1; e >= 0; --e)
      if (VT::get(g_word, e) == g.v) found = g_v0 + e;
    g.idx = found;
    g_v0 = INT_MAX;
  }

  // kN 16-byte vectors; vector u holds entries v_of[u] .., v_of[u] ==
  // INT_MAX marks a padding vector (-inf entries), which adds nothing.
  // kAnyOrder: the thread's vectors may come in any order of their indices
  // (t = 0 then compares indices at a tie), else in increasing order.
  template <int kN, bool kAnyOrder = false>
  __device__ __forceinline__ void tile(const uint4 (&w)[kN], const int (&v_of)[kN], float c2) {
    using VT = Vec<T>;
    constexpr int VEC = VT::N;
    float wm[kN];
    float tm = -INFINITY;
#pragma unroll
    for (int u = 0; u < kN; ++u) {
      wm[u] = VT::vmax(w[u]);
      tm = fmax_nan(tm, wm[u]);
    }
    if (tm != tm) {
      flags |= 1;
      return;
    }
    if (kGreedy) {
      // vectors arrive in increasing index order: the strict > keeps the
      // first vector that reaches the maximum
#pragma unroll
      for (int u = 0; u < kN; ++u) {
        const bool earlier_tie = kAnyOrder && wm[u] == g.v && v_of[u] < (g_v0 != INT_MAX ? g_v0 : g.idx);
        if (v_of[u] != INT_MAX && (g.idx == INT_MAX || wm[u] > g.v || earlier_tie)) {
          g.v = wm[u];
          g_word = w[u];
          g_v0 = v_of[u];
          g.idx = INT_MAX - 1;  // resolved by finalize()
        }
      }
    } else {
      if (tm == INFINITY) flags |= 1;
      if (tm > st.m) {
        const float M2n = tm * c2;
        st.s = st.s * exp2f(M2 - M2n);
        st.m = tm;
        M2 = M2n;
      }
      if (st.m != -INFINITY) {
        // packed fp32 pairs: one FFMA2 and one FADD2 per two entries
        const float2 c2v = make_float2(c2, c2), nM2 = make_float2(-M2, -M2);
        float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
        for (int u = 0; u < kN; ++u) {
#pragma unroll
          for (int e = 0; e < VEC; e += 2) {
            const float2 y = __ffma2_rn(make_float2(VT::get(w[u], e), VT::get(w[u], e + 1)), c2v, nM2);
            const float2 ex = make_float2(ex2_approx(y.x), ex2_approx(y.y));
            if ((e >> 1) & 1) acc1 = __fadd2_rn(acc1, ex);
            else acc0 = __fadd2_rn(acc0, ex);
          }
        }
        st.s += (acc0.x + acc0.y) + (acc1.x + acc1.y);
      }
    }
  }
};

// Streams entries [v0, v1) of `row` into acc with 16-byte loads, kN vectors
// in flight per thread of the kThreads of the CTA (any alignment: a scalar
// head and tail around the aligned body).  Indices reported to acc are
// v + vofs (a shard's first column, or 0).
//
// kFold: vectors past the last whole round, if at most one per thread, are
// loaded with the first round (a ninth vector for some threads) instead of
// making a round trip of their own at the end.
template <typename T, bool kGreedy, int kThreads = kStreamThreads, int kN = kUnroll, bool kFold = false>
__device__ __forceinline__ void stream_chunk(RowAcc<T, kGreedy>& acc, const T* row, int v0, int v1, int vofs,
                                             float c2) {
  using VT = Vec<T>;
  constexpr int VEC = VT::N;
  const uintptr_t addr = reinterpret_cast<uintptr_t>(row + v0);
  const int head = min((int)(((16u - (unsigned)(addr & 15u)) & 15u) / sizeof(T)), v1 - v0);
  const int body0 = v0 + head;
  const int nvec = (v1 - body0) / VEC;
  const int tail0 = body0 + nvec * VEC;
  // head: elements before the first 16-byte boundary (lowest indices)
  if ((int)threadIdx.x < head) acc.scalar(vofs + v0 + threadIdx.x, load_elem(row + v0 + threadIdx.x), c2);
  // body: 16-byte vectors
  const uint4* vp = reinterpret_cast<const uint4*>(row + body0);
  int nround = nvec;  // vectors taken in whole-round steps
  uint4 xw[1] = {make_uint4(VT::kPad, VT::kPad, VT::kPad, VT::kPad)};
  int xv[1] = {INT_MAX};
  if (kFold) {
    const int rem = nvec % (kThreads * kN);
    if (rem != 0 && rem <= kThreads && nvec > rem) {
      nround = nvec - rem;
      if ((int)threadIdx.x < rem) {
        xw[0] = ldg_stream(vp + nround + threadIdx.x);
        xv[0] = vofs + body0 + (nround + threadIdx.x) * VEC;
      }
    }
  }
  for (int base = threadIdx.x; base < nround; base += kThreads * kN) {
    uint4 w[kN];
    int v_of[kN];
#pragma unroll
    for (int u = 0; u < kN; ++u) {
      const int vi = base + u * kThreads;
      w[u] = vi < nround ? ldg_stream(vp + vi) : make_uint4(VT::kPad, VT::kPad, VT::kPad, VT::kPad);
      v_of[u] = vi < nround ? vofs + body0 + vi * VEC : INT_MAX;
    }
    acc.template tile<kN, kFold>(w, v_of, c2);
    if (kFold && base == (int)threadIdx.x) acc.template tile<1, true>(xw, xv, c2);
  }
  // tail: the last < VEC elements (highest indices)
  if (tail0 + (int)threadIdx.x < v1) acc.scalar(vofs + tail0 + threadIdx.x, load_elem(row + tail0 + threadIdx.x), c2);
}

// The CTA's (kThreads threads) reduction of a streamed chunk into one
// partial, valid in thread 0.  Every thread of the CTA calls it.
template <typename T, bool kGreedy, int kThreads = kStreamThreads>
__device__ __forceinline__ RowPartial cta_reduce_partial(RowAcc<T, kGreedy>& acc, float c2) {
  __shared__ float sh_a[kThreads / 32];
  __shared__ float sh_b[kThreads / 32];
  __shared__ int32_t sh_i[kThreads / 32];
  __shared__ int32_t sh_f[kThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  acc.finalize();
  const int32_t flags = __reduce_or_sync(0xFFFFFFFFu, (unsigned)acc.flags);
  RowPartial out{0.0f, 0.0f, 0, 0};
  if (kGreedy) {
    ArgState g = acc.g;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      ArgState other{__shfl_xor_sync(0xFFFFFFFFu, g.v, o), __shfl_xor_sync(0xFFFFFFFFu, g.idx, o)};
      if (arg_better(other, g)) g = other;
    }
    if (lane == 0) {
      sh_a[warp] = g.v;
      sh_i[warp] = g.idx;
      sh_f[warp] = flags;
    }
    consumer_sync<kThreads>();
    if (threadIdx.x == 0) {
      ArgState best{sh_a[0], sh_i[0]};
      int32_t f = sh_f[0];
      for (int k = 1; k < kThreads / 32; ++k) {
        ArgState o{sh_a[k], sh_i[k]};
        if (arg_better(o, best)) best = o;
        f |= sh_f[k];
      }
      out.m = best.v;
      out.idx = best.idx;
      out.flags = f;
    }
  } else {
    SoftState st = acc.st;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      SoftState other{__shfl_xor_sync(0xFFFFFFFFu, st.m, o), __shfl_xor_sync(0xFFFFFFFFu, st.s, o)};
      st = soft_merge(st, other, c2);
    }
    if (lane == 0) {
      sh_a[warp] = st.m;
      sh_b[warp] = st.s;
      sh_f[warp] = flags;
    }
    consumer_sync<kThreads>();
    if (threadIdx.x == 0) {
      SoftState all{sh_a[0], sh_b[0]};
      int32_t f = sh_f[0];
      for (int k = 1; k < kThreads / 32; ++k) {
        all = soft_merge(all, SoftState{sh_a[k], sh_b[k]}, c2);
        f |= sh_f[k];
      }
      out.m = all.m;
      out.s = all.s;
      out.flags = f;
    }
  }
  return out;
}

// ---------------------------------------------------------------------------
// Sampling pass (t > 0)
// ---------------------------------------------------------------------------
// Eight consecutive entries of a row as floats, from 16-byte loads: from
// global memory (streaming) or from a chunk staged in shared memory.
template <bool kShared>
__device__ __forceinline__ uint4 load16(const void* ptr) {
  if (kShared) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"((uint32_t)__cvta_generic_to_shared(ptr)));
    return v;
  }
  return ldg_stream(ptr);
}

template <typename T>
struct Row8;
template <>
struct Row8<__nv_bfloat16> {
  template <bool kShared>
  __device__ static void load(const void* row, int g8, float x[8]) {
    const uint4 w = load16<kShared>(static_cast<const uint4*>(row) + g8);
    x[0] = bf16_lo(w.x);
    x[1] = bf16_hi(w.x);
    x[2] = bf16_lo(w.y);
    x[3] = bf16_hi(w.y);
    x[4] = bf16_lo(w.z);
    x[5] = bf16_hi(w.z);
    x[6] = bf16_lo(w.w);
    x[7] = bf16_hi(w.w);
  }
};
template <>
struct Row8<float> {
  template <bool kShared>
  __device__ static void load(const void* row, int g8, float x[8]) {
    const uint4 a = load16<kShared>(static_cast<const uint4*>(row) + 2 * g8);
    const uint4 b = load16<kShared>(static_cast<const uint4*>(row) + 2 * g8 + 1);
    x[0] = __uint_as_float(a.x);
    x[1] = __uint_as_float(a.y);
    x[2] = __uint_as_float(a.z);
    x[3] = __uint_as_float(a.w);
    x[4] = __uint_as_float(b.x);
    x[5] = __uint_as_float(b.y);
    x[6] = __uint_as_float(b.z);
    x[7] = __uint_as_float(b.w);
  }
};

// ---------------------------------------------------------------------------
// Two-level exponential race
// ---------------------------------------------------------------------------
// The draw from weights w is made in two exact steps: the level-1 block
// b* = argmin_{W_b > 0} E_b / W_b over blocks of kRaceBlock consecutive
// entries (W_b = sum_{v in b} w_v), then y = argmin_{v in b*, w_v > 0} E'_v / w_v
// (ties to the lowest index).  Level 1 needs one variate per block, so the
// Philox work is 1/kRaceBlock of a per-entry race, and level 2 touches one
// block.  Block variates use purpose SAMPLE (sub-index b / 4, word b % 4), entry
// variates purpose SAMPLE_IN_BLOCK (sub-index v / 4, word v % 4).
constexpr int kRaceBlock = SPEC_RACE_BLOCK;  // entries per block (one warp step here: 32 lanes x 8)
static_assert(kRaceBlock == 256, "the race kernels take a block as one warp step of 32 lanes x 8 entries");
constexpr int kRaceQuad = 4 * kRaceBlock;    // the four blocks of one Philox call

// Race variate of a Philox word: E = -ln(u), u = (2 * (word >> 9) + 1) * 2^-24.
// With m = 2^24 * (1 - u), an odd integer below 2^24, E = -ln(1 - m * 2^-24).
__device__ __forceinline__ uint32_t race_m(uint32_t word) { return ((word >> 8) & 0xFFFFFEu) ^ 0xFFFFFFu; }

// One race entry with weight w: key E / w.  The filter m < thr24 * w, thr24 =
// 2^24 * (a key already held), skips the logarithm when the entry cannot win
// (E >= 1 - u); a weight of 0 never passes it.  Entries arrive in increasing
// index, so the strict comparison keeps the lowest index on ties.
__device__ __forceinline__ float race_key(uint32_t m, float w) { return -log1pf(-((float)m * 0x1p-24f)) / w; }

__device__ __forceinline__ void race_entry(KeyState& best, float& thr24, float w, uint32_t m, int idx) {
  const float mf = (float)m;
  if (mf < thr24 * w) {
    const float key = race_key(m, w);
    if (key < best.key) {
      best = KeyState{key, idx};
      thr24 = fminf(thr24, key * 0x1p24f);
    }
  }
}

// Weight of entry v in the draw.  Residual: max(0, p - q) (normalised p);
// Excl: p * S with the rejected one-hot draft z_excl removed; P: p * S.  The
// roundings are explicit so that both levels compute identical weights.
enum { kWeightResidual = 0, kWeightExcl = 1, kWeightP = 2 };
template <int kMode>
__device__ __forceinline__ float weight_of(float ew, float qv, int v, float invS, int z_excl) {
  if (kMode == kWeightResidual) return fmaxf(0.0f, __fsub_rn(__fmul_rn(ew, invS), qv));
  if (kMode == kWeightExcl) return v == z_excl ? 0.0f : ew;
  return ew;
}
__device__ __forceinline__ float p_weight(float x, float c2, float M2) {
  return ex2_approx(__fmaf_rn(x, c2, -M2));  // p_v * S
}
template <int kMode>
__device__ __forceinline__ float race_weight(float x, float qv, int v, float c2, float M2, float invS, int z_excl) {
  return weight_of<kMode>(p_weight(x, c2, M2), qv, v, invS, z_excl);
}

struct RaceArgs {
  int z_excl;
  float c2, M2, invS;
  uint32_t position;
  uint64_t req;
  uint32_t k0, k1;
};

// Where level 1 reads a row from (see race_level1_impl).
enum { kSrcGlobalVec = 0, kSrcShared = 1, kSrcGlobalScalar = 2 };

// Raw 16-byte words of lane l's 8 entries of the four blocks of quad q
// (entries 1024q + 256s + 8l .. +7); entries at or past V, and blocks s with
// raced[s] false, are not read.
template <typename E, int kSrc>
struct QuadWords {
  static constexpr int kWords = sizeof(E) == 4 ? 2 : 1;  // 16-byte words per 8 entries
  uint4 w[4][kWords];
  __device__ __forceinline__ void load(const void* base, int q, int V, int base_v, const bool (&raced)[4]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int s = 0; s < 4; ++s) {
      const int v8 = q * kRaceQuad + s * kRaceBlock + 8 * lane;
#pragma unroll
      for (int h = 0; h < kWords; ++h)
        w[s][h] = raced[s] && v8 < V
                      ? load16<kSrc == kSrcShared>(static_cast<const uint4*>(base) + (((v8 - base_v) >> 3) * kWords + h))
                      : make_uint4(0u, 0u, 0u, 0u);
    }
  }
  __device__ __forceinline__ float get(int s, int e) const {
    if (kWords == 2) {
      const uint4& u = w[s][e >> 2];
      const uint32_t x = (e & 3) == 0 ? u.x : (e & 3) == 1 ? u.y : (e & 3) == 2 ? u.z : u.w;
      return __uint_as_float(x);
    }
    const uint4& u = w[s][0];
    const uint32_t x = e < 2 ? u.x : e < 4 ? u.y : e < 6 ? u.z : u.w;
    return (e & 1) ? bf16_hi(x) : bf16_lo(x);
  }
};

// Level 1 over quads [q_first, q_end) of the row, quad q to warp
// (q - q_first) mod nwarps.  Entry indices are those of the whole vocabulary;
// `row` (and `qrow`) address entry base_v, and entries at or past V are not
// read.  One block is one warp step: lane l holds entries 8l..8l+7 of it
// (kSrc 0: 16-byte loads from global memory, the whole quad's loads issued at
// once; kSrc 1: the same from shared memory) or entries l + 32e (kSrc 2:
// scalar loads, any layout).  Every lane computes the same block sum and so
// holds the same best block.
//
// kDual also runs the race with weights p (best_p) on the same block variates:
// the draw a sharded caller falls back to when no shard has a positive weight.
// kRange races only the blocks whose entries all lie in [lo, V), plus the
// vocabulary's last block when tail_whole (V is then the vocabulary's end):
// the blocks a vocabulary shard [lo, V) owns whole.
template <typename T, typename Q, int kMode, int kSrc, bool kDual, bool kRange>
__device__ void race_level1_impl(const void* row, const void* qrow, int q_dtype, int V, int base_v, int q_first,
                                 int q_end, int warp_id, int nwarps, const RaceArgs& a, KeyState& best,
                                 KeyState& best_p, int lo, bool tail_whole) {
  const int lane = threadIdx.x & 31;
  float thr24 = best.key * 0x1p24f;
  float thr24p = kDual ? best_p.key * 0x1p24f : 0.0f;
  for (int q = q_first + warp_id; q < q_end; q += nwarps) {
    bool raced[4];
#pragma unroll
    for (int s = 0; s < 4; ++s) {
      const int vb = q * kRaceQuad + s * kRaceBlock;
      raced[s] = vb < V && (!kRange || (vb >= lo && (tail_whole || vb + kRaceBlock <= V)));
    }
    if (kSrc == kSrcGlobalScalar) {
      const uint4 r = philox(draw_counter(a.position, a.req, SPEC_PURPOSE_SAMPLE, (uint32_t)q), a.k0, a.k1);
      const uint32_t words[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        const int vb = q * kRaceQuad + s * kRaceBlock;
        float wsum = 0.0f, wsum_p = 0.0f;
        if (raced[s]) {
          float x[8], qv[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int v = vb + lane + 32 * e;
            x[e] = v < V ? load_elem(static_cast<const T*>(row) + (v - base_v)) : 0.0f;
            qv[e] = (kMode == kWeightResidual && v < V) ? load_any(qrow, q_dtype, v - base_v) : 0.0f;
          }
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int v = vb + lane + 32 * e;
            if (v < V) {
              const float ew = p_weight(x[e], a.c2, a.M2);
              wsum += weight_of<kMode>(ew, qv[e], v, a.invS, a.z_excl);
              if (kDual) wsum_p += ew;
            }
          }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) wsum += __shfl_xor_sync(0xFFFFFFFFu, wsum, o);
        race_entry(best, thr24, wsum, race_m(words[s]), 4 * q + s);
        if (kDual) {
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) wsum_p += __shfl_xor_sync(0xFFFFFFFFu, wsum_p, o);
          race_entry(best_p, thr24p, wsum_p, race_m(words[s]), 4 * q + s);
        }
      }
    } else {
      QuadWords<T, kSrc> xw;
      QuadWords<Q, kSrc> qw;
      xw.load(row, q, V, base_v, raced);
      if (kMode == kWeightResidual) qw.load(qrow, q, V, base_v, raced);
      const uint4 r = philox(draw_counter(a.position, a.req, SPEC_PURPOSE_SAMPLE, (uint32_t)q), a.k0, a.k1);
      const uint32_t words[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        const int v8 = q * kRaceQuad + s * kRaceBlock + 8 * lane;
        float wsum = 0.0f, wsum_p = 0.0f;
        if (raced[s] && v8 < V) {
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float ew = p_weight(xw.get(s, e), a.c2, a.M2);
            wsum += weight_of<kMode>(ew, kMode == kWeightResidual ? qw.get(s, e) : 0.0f, v8 + e, a.invS, a.z_excl);
            if (kDual) wsum_p += ew;
          }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) wsum += __shfl_xor_sync(0xFFFFFFFFu, wsum, o);
        race_entry(best, thr24, wsum, race_m(words[s]), 4 * q + s);
        if (kDual) {
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) wsum_p += __shfl_xor_sync(0xFFFFFFFFu, wsum_p, o);
          race_entry(best_p, thr24p, wsum_p, race_m(words[s]), 4 * q + s);
        }
      }
    }
  }
}

template <typename T, typename Q, int kMode, int kSrc>
__device__ __forceinline__ void race_level1(const void* row, const void* qrow, int q_dtype, int V, int base_v,
                                            int q_first, int q_end, int warp_id, int nwarps, const RaceArgs& a,
                                            KeyState& best) {
  race_level1_impl<T, Q, kMode, kSrc, false, false>(row, qrow, q_dtype, V, base_v, q_first, q_end, warp_id, nwarps, a,
                                                    best, best, 0, true);
}

// Minimum key over the CTA (valid in thread 0).  sh: kSampleThreads / 32 slots.
__device__ __forceinline__ KeyState cta_min_key(KeyState b, KeyState* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    KeyState other{__shfl_xor_sync(0xFFFFFFFFu, b.key, o), __shfl_xor_sync(0xFFFFFFFFu, b.idx, o)};
    if (key_better(other, b)) b = other;
  }
  if (lane == 0) sh[warp] = b;
  __syncthreads();
  if (threadIdx.x == 0)
    for (int k = 0; k < kSampleThreads / 32; ++k)
      if (key_better(sh[k], b)) b = sh[k];
  __syncthreads();
  return b;
}

// Level 2 in block b (one entry per thread; result in thread 0).
template <typename T, int kMode>
__device__ KeyState race_level2(const T* row, const void* qrow, int q_dtype, int V, int base_v, int b, const RaceArgs& a,
                                KeyState* sh) {
  const int v = b * kRaceBlock + (int)threadIdx.x;
  KeyState best{INFINITY, INT_MAX};
  if (v < V) {
    const float x = load_elem(row + (v - base_v));
    const float qv = kMode == kWeightResidual ? load_any(qrow, q_dtype, v - base_v) : 0.0f;
    const float w = race_weight<kMode>(x, qv, v, a.c2, a.M2, a.invS, a.z_excl);
    const uint4 r = philox(draw_counter(a.position, a.req, SPEC_PURPOSE_SAMPLE_IN_BLOCK, (uint32_t)(v >> 2)), a.k0,
                           a.k1);
    const uint32_t word = (v & 3) == 0 ? r.x : (v & 3) == 1 ? r.y : (v & 3) == 2 ? r.z : r.w;
    if (w > 0.0f) best = KeyState{race_key(race_m(word), w), v};
  }
  return cta_min_key(best, sh);
}

// Level 1 of this CTA's part of the row, dispatched on the weight mode, the
// q element type and the layout (16-byte loads need V % 8 == 0 and aligned
// rows).
template <typename T, int kMode>
__device__ void race_level1_any(const VerifyLaunch& p, const void* row, const void* qrow, int q_first, int q_end,
                                int warp_id, int nwarps, const RaceArgs& a, KeyState& best) {
  if (p.vec_s) {
    if (kMode == kWeightResidual && p.q_dtype == SPEC_F32)
      race_level1<T, float, kMode, kSrcGlobalVec>(row, qrow, p.q_dtype, p.V, 0, q_first, q_end, warp_id, nwarps, a,
                                                  best);
    else
      race_level1<T, __nv_bfloat16, kMode, kSrcGlobalVec>(row, qrow, p.q_dtype, p.V, 0, q_first, q_end, warp_id,
                                                          nwarps, a, best);
  } else {
    race_level1<T, T, kMode, kSrcGlobalScalar>(row, qrow, p.q_dtype, p.V, 0, q_first, q_end, warp_id, nwarps, a,
                                               best);
  }
}


// ---------------------------------------------------------------------------
// Request shape and the decision chain
// ---------------------------------------------------------------------------
// Shape of request i as the streaming CTAs see it: every CTA of the request
// reads the same header, so all agree on n and on the arrival target.  A
// request whose header is inconsistent streams nothing; its (row 0, chunk 0)
// CTA alone arrives and reports it.
struct ReqShape {
  int n;
  long long row0;
  bool valid;
};

// kL2: load through L2 only (loads a kernel issues before its grid-dependency
// wait, of data that kernels before the previous one wrote).
template <bool kL2, typename E>
__device__ __forceinline__ E load_in(const E* a) {
  return kL2 ? __ldcg(a) : __ldg(a);
}

template <class L, bool kL2 = false>
__device__ __forceinline__ ReqShape request_shape(const L& p, int i) {
  const int n_in = p.depth ? load_in<kL2>(p.depth + i) : p.K;
  long long off0 = (long long)i * (p.K + 1), off1 = off0 + n_in + 1;
  if (p.row_offsets) {
    off0 = load_in<kL2>(p.row_offsets + i);
    off1 = load_in<kL2>(p.row_offsets + i + 1);
  }
  const long long pos = load_in<kL2>(reinterpret_cast<const long long*>(p.pos_base) + i);
  ReqShape s;
  s.valid = n_in >= 0 && n_in <= p.K && off0 >= 0 && off1 == off0 + n_in + 1 && off1 <= p.R_max &&
            pos >= 0 && pos + n_in <= 0xFFFFFFFFLL;
  s.n = s.valid ? n_in : 0;
  s.row0 = s.valid ? off0 : 0;
  return s;
}

// What a decision needs that the rows' statistics do not decide: seeds,
// draft tokens and (kDraws) the acceptance variates, prepared by the deciding
// warp before the statistics are complete (before the arrival atomic, or
// before the grid-dependency wait).  z[u] and u[u] belong to draft
// j = lane + 32u.
struct DecidePre {
  uint32_t pos;
  unsigned long long seed, req;
  int32_t z[(kMaxRows + 31) / 32];
  float u[(kMaxRows + 31) / 32];
};
template <class L, bool kL2 = false, bool kDraws = false>
__device__ __forceinline__ DecidePre decide_prefetch(const L& p, int i) {
  const int lane = threadIdx.x & 31;
  DecidePre pre;
  pre.pos = (uint32_t)load_in<kL2>(reinterpret_cast<const long long*>(p.pos_base) + i);
  pre.seed = load_in<kL2>(reinterpret_cast<const unsigned long long*>(p.seeds) + i);
  pre.req = load_in<kL2>(reinterpret_cast<const unsigned long long*>(p.request_ids) + i);
#pragma unroll
  for (int u = 0; u < (kMaxRows + 31) / 32; ++u) {
    const int j = lane + 32 * u;
    pre.z[u] = j < p.K ? load_in<kL2>(p.drafts + (size_t)i * p.K + j) : 0;
    pre.u[u] = 1.0f;
    if (kDraws && j < p.K) {
      // u_j, the uniform of draft j's acceptance test: 24 bits, exactly
      const uint4 w = philox(draw_counter(pre.pos + (uint32_t)j, pre.req, SPEC_PURPOSE_ACCEPT, 0u),
                             (uint32_t)pre.seed, (uint32_t)(pre.seed >> 32));
      pre.u[u] = (float)(w.x >> 8) * 0x1p-24f;
    }
  }
  return pre;
}

// The decision chain of request i, one warp, once the rows' statistics are
// gathered: sh_m / sh_S (t > 0) or sh_m / sh_g (t = 0) per row, sh_z the draft
// tokens, lz / qz (t > 0) the target logit and the draft probability at each
// lane's drafts (draft j = lane + 32u), bad = input error already seen.
// Tests every kept draft, writes the committed prefix, p(z) and the row
// statistics, and either the argmax token (t = 0) or the record of the row to
// sample (t > 0).  The arithmetic is fp32: p_j(z) = 2^(l_z*c2 - fl(m*c2)) / S
// carries a relative error of a few 1e-7, inside the 1e-5 tolerance on
// probabilities, and an acceptance decision can move only where
// |u - min(1, p/q)| is of that order.
struct DecideArrays {
  float* m;
  float* S;
  int32_t* g;
  int32_t* z;
  float* pz;
};

// `outputs`: write the request's outputs (several CTAs may run the same
// decision; one of them writes); `rec_dst` (t > 0): where the record of the
// row to sample goes.
// The decision's outputs, one warp, from the decision arrays (sh.z the
// drafts, sh.pz p_j(z), sh.m / sh.S or sh.m the row statistics): the
// committed prefix (the sampled or argmax token at position a is written
// apart), -1 past it, a, p(z) and the row statistics; for a flagged request
// -1 tokens, a = 0 and zero probabilities.
template <bool kGreedy, class L>
__device__ __forceinline__ void write_decision(const L& p, int i, const ReqShape& rs, const DecideArrays& sh, int a,
                                               int bad) {
  const int K = p.K, n = rs.n;
  const int lane = threadIdx.x & 31;
  int32_t* tok = p.out_tokens + (size_t)i * (K + 1);
  if (bad) {
    if (lane == 0) report(p.status, SPEC_ERR_BAD_INPUT);
    for (int j = lane; j <= K; j += 32) tok[j] = -1;
    if (lane == 0) p.accepted_len[i] = 0;
    if (p.p_draft)
      for (int j = lane; j < K; j += 32) p.p_draft[(size_t)i * K + j] = 0.0f;
    return;
  }
  for (int j = lane; j <= K; j += 32) {
    if (j < a) tok[j] = sh.z[j];
    else if (j > a) tok[j] = -1;
  }
  if (lane == 0) p.accepted_len[i] = a;
  if (p.p_draft)
    for (int j = lane; j < K; j += 32) p.p_draft[(size_t)i * K + j] = j < n ? sh.pz[j] : 0.0f;
  if (p.row_stats) {
    for (int j = lane; j <= n; j += 32) {
      float2 st;
      if (kGreedy) {
        st = make_float2(sh.m[j], 0.0f);
      } else {
        // ln S relative to the exact max / t: S is kept relative to
        // fl(m * c2), and fmaf gives m * c2 - fl(m * c2) exactly
        const float c2 = p.c2;
        const float resid = fmaf(sh.m[j], c2, -(sh.m[j] * c2));
        st = make_float2(sh.m[j] * p.inv_t, (log2f(sh.S[j]) - resid) * 0.69314718055994531f);
      }
      reinterpret_cast<float2*>(p.row_stats)[rs.row0 + j] = st;
    }
  }
}

template <bool kGreedy, class L>
__device__ __forceinline__ void decide_chain(const L& p, int i, const ReqShape& rs, const DecidePre& pre,
                                             const DecideArrays& sh, const float (&lz)[(kMaxRows + 31) / 32],
                                             const float (&qz)[(kMaxRows + 31) / 32], int bad, bool outputs,
                                             ReqRec* rec_dst) {
  const int K = p.K;
  const float c2 = p.c2;
  const int lane = threadIdx.x & 31;
  const int n = rs.n;
  const long long row0 = rs.row0;
  const uint32_t pos = pre.pos;
  float* sh_m = sh.m;
  float* sh_S = sh.S;
  int32_t* sh_g = sh.g;
  int32_t* sh_z = sh.z;
  float* sh_pz = sh.pz;
  // ---- acceptance test of every kept draft (a lane per draft) ----
  int first_reject = n;
  if (!bad) {
#pragma unroll
    for (int u = 0; u < (kMaxRows + 31) / 32; ++u) {
      const int j = lane + 32 * u;
      if (j >= n) break;
      const int z = sh_z[j];
      bool reject;
      if (kGreedy) {
        reject = z != sh_g[j];
        sh_pz[j] = reject ? 0.0f : 1.0f;
      } else {
        // l_z * c2 - fl(m * c2) with one rounding
        const float pz = exp2f(fmaf(lz[u], c2, -(sh_m[j] * c2))) / sh_S[j];
        if (p.dense_q && (!(qz[u] >= 0.0f) || isinf(qz[u]))) bad = 1;
        float r;
        if (qz[u] > 0.0f)
          r = fminf(1.0f, pz / qz[u]);
        else
          r = pz > 0.0f ? 1.0f : 0.0f;
        reject = !(pre.u[u] < r);  // u_j drawn by decide_prefetch
        sh_pz[j] = pz;
      }
      if (reject) first_reject = min(first_reject, j);
    }
  }
  bad = __any_sync(0xFFFFFFFFu, bad);
  first_reject = (int)__reduce_min_sync(0xFFFFFFFFu, (unsigned)first_reject);
  __syncwarp();

  const int a = bad ? 0 : first_reject;
  int32_t* tok = p.out_tokens + (size_t)i * (K + 1);
  if (outputs) write_decision<kGreedy>(p, i, rs, sh, a, bad);
  if (lane == 0) {
    if (kGreedy) {
      if (!bad && outputs) tok[a] = sh_g[a];
    } else {
      ReqRec rec;
      rec.a = a;
      rec.flags = (bad ? 1 : 0) | (a < n ? 2 : 0) | (a < n && p.dense_q ? 4 : 0);
      rec.z_excl = (!bad && a < n) ? sh_z[a] : -1;
      rec.position = pos + (uint32_t)a;
      rec.srow = row0 + a;
      rec.M2 = bad ? 0.0f : sh_m[a] * c2;
      rec.invS = bad ? 0.0f : 1.0f / sh_S[a];
      *rec_dst = rec;
    }
  }
  __syncwarp();
}


}  // namespace spec
