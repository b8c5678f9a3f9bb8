// verify.cu -- batched speculative verification on sm_103a.
//
// Two kernels per call (Section 1 of arxiv 2607.25852: the target verifies
// the drafted tokens in one pass by rejection sampling; temperature 0 is the
// longest argmax-matching prefix):
//
//   stream_rows_kernel   one CTA per (packed row, vocabulary chunk).  Streams
//                        the chunk once with 16-byte loads and writes a
//                        16-byte partial: (max, sum of 2^(l*c2 - fl(max*c2)))
//                        at t > 0, (max, lowest argmax) at t = 0.  This is the
//                        HBM-bound pass: every retained logit is read once.
//   decide_sample_kernel one CTA per (request, vocabulary chunk).  Every CTA of
//                        a request merges the row partials of that request
//                        (a few hundred bytes), re-derives the accept/reject
//                        chain (p_j(z_{j+1}) in fp64 from the merged statistics,
//                        one Philox draw per draft) and then streams its chunk
//                        of the single row that is sampled (residual row at
//                        the first rejection, else the bonus row), running the
//                        exponential race y = argmin E_v / w_v.  The last CTA
//                        of the request to finish (atomic arrival counter,
//                        no spinning) merges the race partials and writes y.
//
// Nothing in the data path waits on another CTA: cross-CTA combination goes
// through a kernel boundary (rows) or a last-arrival counter (race).
#include <float.h>
#include <math.h>

#include <algorithm>

#include "spec_internal.cuh"

namespace spec {

constexpr int kStreamThreads = 256;
constexpr int kUnroll = 4;
constexpr int kSampleThreads = 256;
constexpr int kMaxRows = SPEC_MAX_DRAFTS + 1;

static inline long long ceil_div(long long a, long long b) { return (a + b - 1) / b; }
static inline long long round_up(long long a, long long b) { return ceil_div(a, b) * b; }

VerifyGeometry verify_geometry(int B, int K, int V) {
  VerifyGeometry g{};
  const long long R_max = (long long)B * (K + 1);
  // Streaming pass: aim for ~4096 (row, chunk) items of >= 4096 elements.
  long long nc = ceil_div(4096, R_max);
  nc = std::max(1LL, std::min(nc, std::max(1LL, (long long)V / 4096)));
  long long chunk = round_up(ceil_div(V, nc), 8);
  nc = ceil_div(V, chunk);  // every chunk non-empty
  // Sampling pass: aim for ~1024 (request, chunk) items of >= 2048 elements.
  long long ncs = ceil_div(1024, B);
  ncs = std::max(1LL, std::min(ncs, std::max(1LL, (long long)V / 2048)));
  long long chunk_s = round_up(ceil_div(V, ncs), 8);
  ncs = ceil_div(V, chunk_s);
  g.NC = (int)nc;
  g.chunk = (int)chunk;
  g.NCS = (int)ncs;
  g.chunk_s = (int)chunk_s;
  g.row_part_off = 0;
  g.race_part_off = round_up((long long)sizeof(RowPartial) * R_max * nc, 256);
  g.counters_off = g.race_part_off + round_up((long long)sizeof(RacePartial) * B * ncs, 256);
  g.bytes = g.counters_off + round_up(sizeof(uint32_t) * (long long)B, 256);
  return g;
}

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

template <typename T, bool kGreedy>
__global__ void __launch_bounds__(kStreamThreads) stream_rows_kernel(const VerifyLaunch p) {
  using VT = Vec<T>;
  constexpr int VEC = VT::N;
  const int item = blockIdx.x;
  const int r = item / p.NC;
  const int c = item - r * p.NC;
  int R = p.R_max;
  if (p.row_offsets) R = min(max(__ldg(p.row_offsets + p.B), 0), p.R_max);
  if (r >= R) return;

  const T* row = static_cast<const T*>(p.logits) + (size_t)r * (size_t)p.V;
  const int v0 = c * p.chunk;
  const int v1 = min(p.V, v0 + p.chunk);
  const uintptr_t addr = reinterpret_cast<uintptr_t>(row + v0);
  const int head = min((int)(((16u - (unsigned)(addr & 15u)) & 15u) / sizeof(T)), v1 - v0);
  const int body0 = v0 + head;
  const int nvec = (v1 - body0) / VEC;
  const int tail0 = body0 + nvec * VEC;
  const float c2 = p.c2;

  // thread state
  int32_t flags = 0;
  ArgState g{-INFINITY, INT_MAX};
  SoftState st{-INFINITY, 0.0f};
  float M2 = -INFINITY;  // fl(st.m * c2)

  auto consume_scalar = [&](int v, float x) {
    if (x != x) {
      flags |= 1;
      return;
    }
    if (kGreedy) {
      if (g.idx == INT_MAX || x > g.v) {
        g.v = x;
        g.idx = v;
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
  };

  // head: elements before the first 16-byte boundary (lowest indices)
  if ((int)threadIdx.x < head) consume_scalar(v0 + threadIdx.x, load_elem(row + v0 + threadIdx.x));

  // body: 16-byte vectors, kUnroll vectors in flight per thread
  const uint4* vp = reinterpret_cast<const uint4*>(row + body0);
  for (int base = threadIdx.x; base < nvec; base += kStreamThreads * kUnroll) {
    uint4 w[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int vi = base + u * kStreamThreads;
      w[u] = vi < nvec ? ldg_stream(vp + vi) : make_uint4(VT::kPad, VT::kPad, VT::kPad, VT::kPad);
    }
    float tm = VT::vmax(w[0]);
#pragma unroll
    for (int u = 1; u < kUnroll; ++u) tm = fmax_nan(tm, VT::vmax(w[u]));
    if (tm != tm) {
      flags |= 1;
      continue;
    }
    if (kGreedy) {
      if (g.idx == INT_MAX || tm > g.v) {
        // locate the first element equal to the tile max (index order)
        int found = INT_MAX;
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
#pragma unroll
          for (int e = 0; e < VEC; ++e) {
            if (found == INT_MAX && VT::get(w[u], e) == tm)
              found = body0 + (base + u * kStreamThreads) * VEC + e;
          }
        }
        g.v = tm;
        g.idx = found;
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
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
#pragma unroll
          for (int e = 0; e < VEC; ++e) acc[e & 3] += ex2_approx(fmaf(VT::get(w[u], e), c2, -M2));
        }
        st.s += (acc[0] + acc[1]) + (acc[2] + acc[3]);
      }
    }
  }

  // tail: the last < VEC elements (highest indices)
  if (tail0 + (int)threadIdx.x < v1)
    consume_scalar(tail0 + threadIdx.x, load_elem(row + tail0 + threadIdx.x));

  // ---- CTA reduction ----
  __shared__ float sh_a[kStreamThreads / 32];
  __shared__ float sh_b[kStreamThreads / 32];
  __shared__ int32_t sh_i[kStreamThreads / 32];
  __shared__ int32_t sh_f[kStreamThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  flags = __reduce_or_sync(0xFFFFFFFFu, (unsigned)flags);
  if (kGreedy) {
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
    __syncthreads();
    if (threadIdx.x == 0) {
      ArgState best{sh_a[0], sh_i[0]};
      int32_t f = sh_f[0];
      for (int k = 1; k < kStreamThreads / 32; ++k) {
        ArgState o{sh_a[k], sh_i[k]};
        if (arg_better(o, best)) best = o;
        f |= sh_f[k];
      }
      RowPartial out;
      out.m = best.v;
      out.s = 0.0f;
      out.idx = best.idx;
      out.flags = f;
      p.row_part[(size_t)r * p.NC + c] = out;
    }
  } else {
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
    __syncthreads();
    if (threadIdx.x == 0) {
      SoftState acc{sh_a[0], sh_b[0]};
      int32_t f = sh_f[0];
      for (int k = 1; k < kStreamThreads / 32; ++k) {
        acc = soft_merge(acc, SoftState{sh_a[k], sh_b[k]}, c2);
        f |= sh_f[k];
      }
      RowPartial out;
      out.m = acc.m;
      out.s = acc.s;
      out.idx = 0;
      out.flags = f;
      p.row_part[(size_t)r * p.NC + c] = out;
    }
  }
}

// ---------------------------------------------------------------------------
// Decision chain + sampling pass
// ---------------------------------------------------------------------------
// 2^e in double from an exactly known exponent: integer part by scaling, the
// fractional part through exp2f (relative error ~1e-7).
__device__ __forceinline__ double exp2_split(double e) {
  if (e < -1074.0) return 0.0;
  const double ei = floor(e);
  const float f = (float)(e - ei);
  return ldexp((double)exp2f(f), (int)ei);
}

template <typename T, bool kGreedy>
__global__ void __launch_bounds__(kSampleThreads) decide_sample_kernel(const VerifyLaunch p) {
  const int i = blockIdx.x / p.NCS;
  const int cs = blockIdx.x - i * p.NCS;
  const int K = p.K, V = p.V;
  const float c2 = p.c2;

  __shared__ int sh_n, sh_bad, sh_first_reject, sh_last;
  __shared__ long long sh_row0;
  __shared__ uint32_t sh_pos;
  __shared__ float sh_m[kMaxRows];
  __shared__ double sh_S[kMaxRows];
  __shared__ int32_t sh_g[kMaxRows];
  __shared__ float sh_pz[kMaxRows];

  if (threadIdx.x == 0) {
    int n = p.depth ? p.depth[i] : K;
    int bad = 0;
    if (n < 0 || n > K) {
      bad = 1;
      n = 0;
    }
    long long row0 = (long long)i * (K + 1);
    if (p.row_offsets) {
      row0 = p.row_offsets[i];
      const long long row1 = p.row_offsets[i + 1];
      if (row0 < 0 || row1 != row0 + n + 1 || row1 > p.R_max) {
        bad = 1;
        row0 = 0;
        n = 0;
      }
    }
    const long long pos = p.pos_base[i];
    if (pos < 0 || pos + n > 0xFFFFFFFFLL) bad = 1;
    sh_n = n;
    sh_row0 = row0;
    sh_pos = (uint32_t)pos;
    sh_bad = bad;
    sh_first_reject = n;
  }
  __syncthreads();
  const int n = sh_n;
  const long long row0 = sh_row0;

  // ---- merge the streaming partials of rows 0..n (one warp per row) ----
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (!sh_bad) {
    for (int j = warp; j <= n; j += kSampleThreads / 32) {
      const RowPartial* part = p.row_part + (size_t)(row0 + j) * p.NC;
      int32_t f = 0;
      if (kGreedy) {
        ArgState best{-INFINITY, INT_MAX};
        for (int cc = lane; cc < p.NC; cc += 32) {
          const RowPartial rp = part[cc];
          f |= rp.flags;
          ArgState o{rp.m, rp.idx};
          if (arg_better(o, best)) best = o;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          ArgState other{__shfl_xor_sync(0xFFFFFFFFu, best.v, o),
                         __shfl_xor_sync(0xFFFFFFFFu, best.idx, o)};
          if (arg_better(other, best)) best = other;
        }
        f = __reduce_or_sync(0xFFFFFFFFu, (unsigned)f);
        if (lane == 0) {
          sh_m[j] = best.v;
          sh_g[j] = best.idx;
          if (f || best.idx == INT_MAX) atomicOr(&sh_bad, 1);
        }
      } else {
        float m = -INFINITY;
        for (int cc = lane; cc < p.NC; cc += 32) m = fmaxf(m, part[cc].m);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
        const float M2 = m * c2;
        double S = 0.0;
        for (int cc = lane; cc < p.NC; cc += 32) {
          const RowPartial rp = part[cc];
          f |= rp.flags;
          if (rp.m != -INFINITY) S += (double)rp.s * (double)exp2f(rp.m * c2 - M2);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) S += __shfl_xor_sync(0xFFFFFFFFu, S, o);
        f = __reduce_or_sync(0xFFFFFFFFu, (unsigned)f);
        if (lane == 0) {
          sh_m[j] = m;
          sh_S[j] = S;
          if (f || !(m > -INFINITY) || !(S > 0.0) || !isfinite(S)) atomicOr(&sh_bad, 1);
        }
      }
    }
  }
  __syncthreads();

  // ---- acceptance test of every kept draft (one thread per draft) ----
  const uint64_t seed = p.seeds[i];
  const uint64_t req = p.request_ids[i];
  if (!sh_bad) {
    for (int j = threadIdx.x; j < n; j += kSampleThreads) {
      const int z = p.drafts[(size_t)i * K + j];
      if (z < 0 || z >= V) {
        atomicOr(&sh_bad, 1);
        continue;
      }
      bool reject;
      if (kGreedy) {
        reject = z != sh_g[j];
        sh_pz[j] = reject ? 0.0f : 1.0f;
      } else {
        const float lz = load_elem(static_cast<const T*>(p.logits) + (size_t)(row0 + j) * V + z);
        const double e = (double)lz * (double)c2 - (double)(sh_m[j] * c2);
        const double pz = exp2_split(e) / sh_S[j];
        double qz = 1.0;
        if (p.q) {
          qz = (double)load_any(p.q, p.q_dtype, ((int64_t)i * K + j) * (int64_t)V + z);
          if (!(qz >= 0.0) || isinf(qz)) {
            atomicOr(&sh_bad, 1);
            continue;
          }
        }
        double r;
        if (qz > 0.0)
          r = fmin(1.0, pz / qz);
        else
          r = pz > 0.0 ? 1.0 : 0.0;
        const uint4 w = philox(draw_counter(sh_pos + (uint32_t)j, req, SPEC_PURPOSE_ACCEPT, 0u),
                               (uint32_t)seed, (uint32_t)(seed >> 32));
        const double u = (double)(w.x >> 8) * 0x1p-24;
        reject = !(u < r);
        sh_pz[j] = (float)pz;
      }
      if (reject) atomicMin(&sh_first_reject, j);
    }
  }
  __syncthreads();

  const bool bad = sh_bad != 0;
  const int a = bad ? 0 : sh_first_reject;
  const bool rejected = a < n;
  int32_t* tok = p.out_tokens + (size_t)i * (K + 1);

  // ---- outputs owned by chunk 0 of the request ----
  if (cs == 0) {
    if (bad) {
      if (threadIdx.x == 0) report(p.status, SPEC_ERR_BAD_INPUT);
      for (int j = threadIdx.x; j <= K; j += kSampleThreads) tok[j] = -1;
      if (threadIdx.x == 0) p.accepted_len[i] = 0;
      if (p.p_draft)
        for (int j = threadIdx.x; j < K; j += kSampleThreads) p.p_draft[(size_t)i * K + j] = 0.0f;
    } else {
      for (int j = threadIdx.x; j <= K; j += kSampleThreads) {
        if (j < a) tok[j] = p.drafts[(size_t)i * K + j];
        else if (j > a) tok[j] = -1;
      }
      if (threadIdx.x == 0) p.accepted_len[i] = a;
      if (p.p_draft)
        for (int j = threadIdx.x; j < K; j += kSampleThreads)
          p.p_draft[(size_t)i * K + j] = j < n ? sh_pz[j] : 0.0f;
      if (p.row_stats) {
        for (int j = threadIdx.x; j <= n; j += kSampleThreads) {
          float2 rs;
          if (kGreedy) {
            rs = make_float2(sh_m[j], 0.0f);
          } else {
            // ln S relative to the exact max/t (S is kept relative to fl(max*c2))
            const double corr = ((double)(sh_m[j] * c2) - (double)sh_m[j] * (double)c2) * 0.6931471805599453;
            rs = make_float2(sh_m[j] * p.inv_t, (float)(log(sh_S[j]) + corr));
          }
          reinterpret_cast<float2*>(p.row_stats)[row0 + j] = rs;
        }
      }
      if (kGreedy && threadIdx.x == 0) tok[a] = sh_g[a];
    }
  }
  if (kGreedy) return;

  // ---- sampling pass over chunk cs of the row to be sampled ----
  KeyState best_r{INFINITY, INT_MAX};  // residual race (or the bonus race)
  KeyState best_p{INFINITY, INT_MAX};  // race on p, fallback of an empty residual
  if (!bad) {
    const long long srow = row0 + a;
    const T* row = static_cast<const T*>(p.logits) + (size_t)srow * V;
    const float M2 = sh_m[a] * c2;
    const float invS = (float)(1.0 / sh_S[a]);
    const int z_excl = rejected ? p.drafts[(size_t)i * K + a] : -1;
    const bool general_q = rejected && p.q != nullptr;
    const void* qrow = general_q ? (const void*)((const char*)p.q + ((size_t)i * K + a) * (size_t)V *
                                                                       (p.q_dtype == SPEC_F32 ? 4 : 2))
                                 : nullptr;
    const uint32_t position = sh_pos + (uint32_t)a;
    const uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
    const int v0 = cs * p.chunk_s;
    const int v1 = min(V, v0 + p.chunk_s);
    // groups of 4 consecutive entries share one Philox block
    for (int grp = (v0 >> 2) + threadIdx.x; grp * 4 < v1; grp += kSampleThreads) {
      const uint4 rnd = philox(draw_counter(position, req, SPEC_PURPOSE_SAMPLE, (uint32_t)grp), k0, k1);
      const uint32_t words[4] = {rnd.x, rnd.y, rnd.z, rnd.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int v = grp * 4 + e;
        if (v >= v1) break;
        const float x = load_elem(row + v);
        const float ew = ex2_approx(fmaf(x, c2, -M2));  // p_v * S
        const float d = (float)(0xFFFFFFu - (words[e] >> 8)) * 0x1p-24f;  // 1 - U', exact
        if (general_q) {
          const float pv = ew * invS;
          const float qv = load_any(qrow, p.q_dtype, v);
          const float wr = fmaxf(0.0f, pv - qv);
          if (wr > 0.0f && d < best_r.key * wr) {
            const float key = -log1pf(-d) / wr;
            if (key < best_r.key) best_r = KeyState{key, v};
          }
          if (pv > 0.0f && d < best_p.key * pv) {
            const float key = -log1pf(-d) / pv;
            if (key < best_p.key) best_p = KeyState{key, v};
          }
        } else {
          if (ew > 0.0f && d < (v == z_excl ? best_p.key : best_r.key) * ew) {
            const float key = -log1pf(-d) / ew;
            if (v == z_excl) {
              if (key < best_p.key) best_p = KeyState{key, v};
            } else if (key < best_r.key) {
              best_r = KeyState{key, v};
            }
          }
        }
      }
    }
    if (!general_q) {
      // the race on p is the residual race plus the excluded draft token
      if (key_better(best_r, best_p)) best_p = best_r;
    }
  }

  // ---- CTA reduction of the two races ----
  __shared__ KeyState sh_r[kSampleThreads / 32], sh_p[kSampleThreads / 32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    KeyState orr{__shfl_xor_sync(0xFFFFFFFFu, best_r.key, o), __shfl_xor_sync(0xFFFFFFFFu, best_r.idx, o)};
    KeyState op{__shfl_xor_sync(0xFFFFFFFFu, best_p.key, o), __shfl_xor_sync(0xFFFFFFFFu, best_p.idx, o)};
    if (key_better(orr, best_r)) best_r = orr;
    if (key_better(op, best_p)) best_p = op;
  }
  if (lane == 0) {
    sh_r[warp] = best_r;
    sh_p[warp] = best_p;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int k = 1; k < kSampleThreads / 32; ++k) {
      if (key_better(sh_r[k], sh_r[0])) sh_r[0] = sh_r[k];
      if (key_better(sh_p[k], sh_p[0])) sh_p[0] = sh_p[k];
    }
    RacePartial rp;
    rp.key_r = sh_r[0].key;
    rp.idx_r = sh_r[0].idx;
    rp.key_p = sh_p[0].key;
    rp.idx_p = sh_p[0].idx;
    p.race_part[(size_t)i * p.NCS + cs] = rp;
    __threadfence();
    const uint32_t prev = atomicAdd(p.counters + i, 1u);
    sh_last = prev == (uint32_t)(p.NCS - 1);
  }
  __syncthreads();
  if (!sh_last || threadIdx.x != 0) return;

  // ---- last CTA of the request: merge the race partials, write y ----
  __threadfence();
  KeyState r_all{INFINITY, INT_MAX}, p_all{INFINITY, INT_MAX};
  for (int k = 0; k < p.NCS; ++k) {
    const RacePartial* src = p.race_part + (size_t)i * p.NCS + k;
    KeyState kr{__ldcg(&src->key_r), __ldcg(&src->idx_r)};
    KeyState kp{__ldcg(&src->key_p), __ldcg(&src->idx_p)};
    if (key_better(kr, r_all)) r_all = kr;
    if (key_better(kp, p_all)) p_all = kp;
  }
  p.counters[i] = 0u;  // leave the workspace zeroed for the next call
  if (bad) return;
  int y = r_all.idx;
  if (!rejected) y = r_all.idx;                 // bonus: race on p_n
  else if (y == INT_MAX) y = p_all.idx;         // empty residual: draw from p
  if (y == INT_MAX) {
    report(p.status, SPEC_ERR_BAD_INPUT);
    tok[a] = -1;
    p.accepted_len[i] = 0;
    return;
  }
  tok[a] = y;
}

// ---------------------------------------------------------------------------
// Launcher
// ---------------------------------------------------------------------------
template <typename T>
static cudaError_t launch_typed(const VerifyLaunch& p, cudaStream_t stream, cudaEvent_t ev_before,
                                cudaEvent_t ev_after) {
  const bool greedy = p.temperature == 0.0f;
  VerifyLaunch pd = p;
  if (greedy) pd.NCS = 1;  // no sampling pass: one decision CTA per request
  const unsigned grid1 = (unsigned)((long long)p.R_max * p.NC);
  const unsigned grid2 = (unsigned)((long long)p.B * pd.NCS);
  if (ev_before) cudaEventRecord(ev_before, stream);
  if (greedy)
    stream_rows_kernel<T, true><<<grid1, kStreamThreads, 0, stream>>>(p);
  else
    stream_rows_kernel<T, false><<<grid1, kStreamThreads, 0, stream>>>(p);
  cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  if (ev_after) cudaEventRecord(ev_after, stream);
  if (greedy)
    decide_sample_kernel<T, true><<<grid2, kSampleThreads, 0, stream>>>(pd);
  else
    decide_sample_kernel<T, false><<<grid2, kSampleThreads, 0, stream>>>(pd);
  return cudaGetLastError();
}

cudaError_t launch_verify(const VerifyLaunch& p, cudaStream_t stream, cudaEvent_t ev_before,
                          cudaEvent_t ev_after) {
  if (p.logits_dtype == SPEC_F32) return launch_typed<float>(p, stream, ev_before, ev_after);
  return launch_typed<__nv_bfloat16>(p, stream, ev_before, ev_after);
}

}  // namespace spec
