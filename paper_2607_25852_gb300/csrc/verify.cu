// verify.cu -- batched speculative verification on sm_103a.
//
// Two kernels per call (Section 1 of arxiv 2607.25852: the target verifies
// the drafted tokens in one pass by rejection sampling; temperature 0 is the
// longest argmax-matching prefix):
//
//   stream_rows_kernel    one CTA per (request, row, vocabulary chunk).
//                         Streams its chunk once with 16-byte loads and
//                         writes a 16-byte partial: (max, sum of
//                         2^(l*c2 - fl(max*c2))) at t > 0, (max, lowest
//                         argmax) at t = 0, and at t > 0 the target logit and
//                         q at the row's draft token if its chunk holds it.
//                         This is the HBM-bound pass: every retained logit is
//                         read once.
//   sample_kernel         t > 0: one CTA per (request, vocabulary chunk) of
//                         the single row that is sampled.  Each CTA first
//                         runs the request's decision chain (merged row
//                         statistics, p_j(z_{j+1}), one Philox uniform per
//                         draft, the first rejection): the residual row at the
//                         first rejection, else the bonus row, is sampled by
//                         the exponential race y = argmin E_v / w_v.  The last
//                         CTA of the request to finish merges the race
//                         partials, draws inside the winning block and writes
//                         the outputs.
//   greedy_decide_kernel  t = 0: one warp per request, the argmax chain.
//
// Nothing waits on another CTA: cross-CTA combination goes through arrival
// counters (the last to arrive does the merge) or the kernel boundary.
#include <float.h>
#include <math.h>

#include <algorithm>

#include "verify_common.cuh"

namespace spec {


static inline long long ceil_div(long long a, long long b) { return (a + b - 1) / b; }
static inline long long round_up(long long a, long long b) { return ceil_div(a, b) * b; }

VerifyGeometry verify_geometry(int B, int K, int V) {
  VerifyGeometry g{};
  const long long R_max = (long long)B * (K + 1);
  // Streaming pass: aim for ~4096 (row, chunk) items, each a whole number of
  // load rounds (256 threads x 8 16-byte vectors = 16384 bf16 entries), so
  // that only the last chunk of a row ends in a partial round.
  long long nc = ceil_div(4096, R_max);
  nc = std::max(1LL, std::min(nc, std::max(1LL, (long long)V / 16384)));
  long long chunk = round_up(ceil_div(V, nc), 16384);
  nc = ceil_div(V, chunk);  // every chunk non-empty
  // Sampling pass: aim for ~560 (request, chunk) CTAs, about one resident
  // wave on 152 SMs, of >= 2048 elements each, every chunk a whole number of
  // race quads (1024 entries).
  long long ncs = ceil_div(560, B);
  ncs = std::max(1LL, std::min(ncs, std::max(1LL, (long long)V / 2048)));
  long long chunk_s = round_up(ceil_div(V, ncs), 1024);
  ncs = ceil_div(V, chunk_s);
  g.NC = (int)nc;
  g.chunk = (int)chunk;
  g.NCS = (int)ncs;
  g.chunk_s = (int)chunk_s;
  g.row_part_off = 0;
  g.race_part_off = round_up((long long)sizeof(RowPartial) * R_max * nc, 256);
  g.view_off = g.race_part_off + round_up((long long)sizeof(RacePartial) * B * ncs, 256);
  // zero region: the sampling pass's arrivals [B]
  g.counters_off = g.view_off + round_up((long long)sizeof(float2) * R_max, 256);
  g.bytes = g.counters_off + round_up(sizeof(uint32_t) * (long long)B, 256);
  return g;
}

// ---------------------------------------------------------------------------
// Decision chain (every sampling CTA at t > 0; greedy_decide_kernel at t = 0)
// ---------------------------------------------------------------------------
// One warp.  Merges the chunk partials of rows 0..n (a lane per row), loads
// the target logit and the draft probability at each draft, and runs the
// decision chain.  Only one warp of a CTA decides at a time: the decision
// arrays (row statistics, drafts, p_j(z)) are per CTA, and are kept after the
// decision for the outputs written later.
__shared__ float sh_m[kMaxRows];
__shared__ float sh_S[kMaxRows];
__shared__ int32_t sh_g[kMaxRows];
__shared__ int32_t sh_z[kMaxRows];
__shared__ float sh_pz[kMaxRows];
__device__ __forceinline__ DecideArrays decide_arrays() { return DecideArrays{sh_m, sh_S, sh_g, sh_z, sh_pz}; }

template <typename T, bool kGreedy>
__device__ __forceinline__ void decide_request(const VerifyLaunch& p, int i, ReqShape rs, const DecidePre& pre,
                                            bool outputs, ReqRec* rec_dst) {
  const int K = p.K, V = p.V, NC = p.NC;
  const float c2 = p.c2;
  const int lane = threadIdx.x & 31;
  const int n = rs.n;
  const long long row0 = rs.row0;

  // ---- one round trip: the row partials (a lane per row), at t > 0 each
  // row's (target logit, q) at its draft from the streaming pass, and the
  // draft tokens (prefetched by the caller) ----
  int bad = rs.valid ? 0 : 1;
  float lz[(kMaxRows + 31) / 32], qz[(kMaxRows + 31) / 32];
#pragma unroll
  for (int u = 0; u < (kMaxRows + 31) / 32; ++u) {
    const int j = lane + 32 * u;
    lz[u] = 0.0f;
    qz[u] = 1.0f;
    if (!kGreedy && rs.valid && j < n) {
      const float2 v = __ldcg(p.draft_view + row0 + j);
      lz[u] = v.x;
      qz[u] = v.y;
    }
  }
  if (rs.valid) {
    for (int j = lane; j <= n; j += 32) {
      const RowPartial* part = p.row_part + (size_t)(row0 + j) * NC;
      int32_t f = 0;
      // kBatch partials in flight per lane
      constexpr int kBatch = 8;
      if (kGreedy) {
        ArgState best{-INFINITY, INT_MAX};
        for (int c0 = 0; c0 < NC; c0 += kBatch) {
          RowPartial rb[kBatch];
#pragma unroll
          for (int u = 0; u < kBatch; ++u)
            if (c0 + u < NC) rb[u] = load_partial_cg(part + c0 + u);
#pragma unroll
          for (int u = 0; u < kBatch; ++u) {
            if (c0 + u >= NC) break;
            f |= rb[u].flags;
            ArgState o{rb[u].m, rb[u].idx};
            if (arg_better(o, best)) best = o;
          }
        }
        sh_m[j] = best.v;
        sh_g[j] = best.idx;
        if (f || best.idx == INT_MAX) bad = 1;
      } else {
        SoftState all{-INFINITY, 0.0f};
        for (int c0 = 0; c0 < NC; c0 += kBatch) {
          RowPartial rb[kBatch];
#pragma unroll
          for (int u = 0; u < kBatch; ++u)
            if (c0 + u < NC) rb[u] = load_partial_cg(part + c0 + u);
#pragma unroll
          for (int u = 0; u < kBatch; ++u) {
            if (c0 + u >= NC) break;
            f |= rb[u].flags;
            all = soft_merge(all, SoftState{rb[u].m, rb[u].s}, c2);
          }
        }
        sh_m[j] = all.m;
        sh_S[j] = all.s;
        if (f || !(all.m > -INFINITY) || !(all.s > 0.0f) || !isfinite(all.s)) bad = 1;
      }
    }
  }
#pragma unroll
  for (int u = 0; u < (kMaxRows + 31) / 32; ++u)
    if (lane + 32 * u < K) sh_z[lane + 32 * u] = pre.z[u];
  __syncwarp();
  for (int j = lane; j < n; j += 32)
    if (sh_z[j] < 0 || sh_z[j] >= V) bad = 1;
  bad = __any_sync(0xFFFFFFFFu, bad);
  __syncwarp();
  decide_chain<kGreedy>(p, i, rs, pre, decide_arrays(), lz, qz, bad, outputs, rec_dst);
  __syncwarp();
}

// End of one (request, row, chunk) item, all threads of the CTA: the CTA
// reduction and the chunk partial (valid requests).  The kernel after this
// one, which waits for this grid anyway, decides each request from the
// complete partials (the sampling kernel at t > 0, greedy_decide_kernel at
// t = 0), so a streaming CTA ends with its partial and holds no SM slot for
// a round trip.
template <typename T, bool kGreedy>
__device__ __forceinline__ void finish_item(const VerifyLaunch& p, RowAcc<T, kGreedy>& acc, const ReqShape& rs,
                                            long long r, int c) {
  if (rs.valid) {
    const RowPartial out = cta_reduce_partial<T, kGreedy>(acc, p.c2);
    if (threadIdx.x == 0) p.row_part[(size_t)r * p.NC + c] = out;
  }
}

// Item of CTA blockIdx.x: (request i, row j, chunk c), request-major, so
// that the requests complete (and are decided) in order.
struct StreamItem {
  int i, j, c;
};
__device__ __forceinline__ StreamItem stream_item(const VerifyLaunch& p) {
  const int per_req = (p.K + 1) * p.NC;
  StreamItem it;
  it.i = blockIdx.x / per_req;
  const int rem = blockIdx.x - it.i * per_req;
  it.j = rem / p.NC;
  it.c = rem - it.j * p.NC;
  return it;
}

// Streaming pass with 16-byte loads from global memory (any alignment: a
// scalar head and tail around the aligned body).
template <typename T, bool kGreedy>
__global__ void __launch_bounds__(kStreamThreads, kGreedy ? 4 : 0) stream_rows_kernel(const VerifyLaunch p) {
  const StreamItem it = stream_item(p);
  pdl_wait_prerequisites();  // row offsets and depths come from the allocator
  const ReqShape rs = request_shape(p, it.i);
  if (!(rs.valid ? it.j <= rs.n : (it.j == 0 && it.c == 0))) return;
  // The sampling kernel may start launching once every CTA here has started;
  // it waits for this grid's completion before it reads anything.
  pdl_launch_dependents();
  RowAcc<T, kGreedy> acc;
  const long long r = rs.row0 + it.j;
  if (rs.valid) {
    const T* row = static_cast<const T*>(p.logits) + (size_t)r * (size_t)p.V;
    const int v0 = it.c * p.chunk;
    const int v1 = min(p.V, v0 + p.chunk);
    // t > 0: the row's draft token, loaded while the chunk streams; the CTA
    // whose chunk holds it records the target logit and q there for the
    // decision (a draft outside [0, V) is left to the decision to report)
    int z = -1;
    if (!kGreedy && threadIdx.x == 0 && it.j < rs.n) z = __ldg(p.drafts + (size_t)it.i * p.K + it.j);
    stream_chunk<T, kGreedy>(acc, row, v0, v1, 0, p.c2);
    if (!kGreedy && threadIdx.x == 0 && z >= v0 && z < v1) {
      const float lz = load_elem(row + z);
      const float qz = p.q ? load_any(p.q, p.q_dtype, ((int64_t)it.i * p.K + it.j) * (int64_t)p.V + z) : 1.0f;
      p.draft_view[r] = make_float2(lz, qz);
    }
  }
  finish_item<T, kGreedy>(p, acc, rs, r, it.c);
}

// t = 0: each request's decision, one warp (one CTA) per request, once the
// streaming kernel has written every row's (max, lowest argmax) partials.
// The request's shape and drafts are the allocator's and the caller's, loaded
// (through L2) while the streaming kernel drains.
template <typename T>
__global__ void __launch_bounds__(32) greedy_decide_kernel(const VerifyLaunch p) {
  const int i = blockIdx.x;
  const ReqShape rs = request_shape<VerifyLaunch, true>(p, i);
  const DecidePre pre = decide_prefetch<VerifyLaunch, true, false>(p, i);
  pdl_wait_prerequisites();  // the row partials of the streaming kernel
  pdl_launch_dependents();   // the commit kernel waits for this grid in turn
  decide_request<T, true>(p, i, rs, pre, true, nullptr);
}

template <typename T>
__global__ void __launch_bounds__(kSampleThreads, 4) sample_kernel(const VerifyLaunch p) {
  __shared__ int sh_last, sh_b;
  __shared__ KeyState sh_red[kSampleThreads / 32];
  const int i = blockIdx.x / p.NCS;
  const int cs = blockIdx.x - i * p.NCS;
  const int V = p.V;
  const int warp = threadIdx.x >> 5;
  __shared__ ReqRec sh_rec;
  // The request's shape, its drafts and seeds and the acceptance variates do
  // not depend on the streaming kernel: they are loaded (through L2) and drawn
  // while it drains.  Their producers completed before this grid could
  // launch: the allocator (the streaming CTAs waited for it before they let
  // this grid start) and the caller's earlier work.
  const ReqShape rs = request_shape<VerifyLaunch, true>(p, i);
  DecidePre pre{};
  if (warp == 0) pre = decide_prefetch<VerifyLaunch, true, true>(p, i);
  pdl_wait_prerequisites();  // the row partials of the streaming kernel
  pdl_launch_dependents();   // the commit kernel waits for this grid in turn
  // The request's decision chain (every CTA of the request runs it; the last
  // CTA to finish the race writes the outputs): which row to sample, and how.
  if (warp == 0) decide_request<T, false>(p, i, rs, pre, false, &sh_rec);
  __syncthreads();
  const ReqRec rec = sh_rec;
  if (rec.flags & 1) {  // bad input: chunk 0 writes the flagged outputs
    if (cs == 0 && warp == 0) write_decision<false>(p, i, rs, decide_arrays(), 0, 1);
    return;
  }
  // A record that could not come from a consistent decision is refused
  // rather than used to read outside the inputs.
  if (rec.a < 0 || rec.a > p.K || rec.srow < 0 || rec.srow >= p.R_max || rec.z_excl < -1 || rec.z_excl >= V ||
      ((rec.flags & 4) && (p.q == nullptr || rec.a >= p.K))) {
    if (threadIdx.x == 0) report(p.status, SPEC_ERR_WORKSPACE);
    return;
  }

  RaceArgs ra;
  ra.z_excl = rec.z_excl;
  ra.c2 = p.c2;
  ra.M2 = rec.M2;
  ra.invS = rec.invS;
  ra.position = rec.position;
  ra.req = __ldg(reinterpret_cast<const unsigned long long*>(p.request_ids) + i);
  const uint64_t seed = __ldg(reinterpret_cast<const unsigned long long*>(p.seeds) + i);
  ra.k0 = (uint32_t)seed;
  ra.k1 = (uint32_t)(seed >> 32);
  // Residual against a dense q at a rejection; p without the draft at a
  // one-hot rejection; p at the bonus row.
  const int mode = (rec.flags & 4) ? kWeightResidual : (rec.flags & 2) ? kWeightExcl : kWeightP;
  const T* row = static_cast<const T*>(p.logits) + (size_t)rec.srow * V;
  const size_t qsize = p.q_dtype == SPEC_F32 ? 4 : 2;
  const void* qrow = mode == kWeightResidual
                         ? (const void*)((const char*)p.q + ((size_t)i * p.K + rec.a) * (size_t)V * qsize)
                         : nullptr;

  // ---- level 1 over this CTA's chunk (whole quads) ----
  const int v0 = cs * p.chunk_s;
  const int v1 = min(V, v0 + p.chunk_s);
  const int q_first = v0 / kRaceQuad;
  const int q_end = (v1 + kRaceQuad - 1) / kRaceQuad;
  KeyState best{INFINITY, INT_MAX};
  if (mode == kWeightResidual)
    race_level1_any<T, kWeightResidual>(p, row, qrow, q_first, q_end, warp, kSampleThreads / 32, ra, best);
  else if (mode == kWeightExcl)
    race_level1_any<T, kWeightExcl>(p, row, qrow, q_first, q_end, warp, kSampleThreads / 32, ra, best);
  else
    race_level1_any<T, kWeightP>(p, row, qrow, q_first, q_end, warp, kSampleThreads / 32, ra, best);

  // ---- CTA reduction; the last CTA of the request to arrive goes on ----
  best = cta_min_key(best, sh_red);
  if (threadIdx.x == 0) {
    RacePartial rp;
    rp.key_r = best.key;
    rp.idx_r = best.idx;
    rp.key_p = INFINITY;
    rp.idx_p = INT_MAX;
    p.race_part[(size_t)i * p.NCS + cs] = rp;
    __threadfence();
    sh_last = atomicAdd(p.counters + i, 1u) == (uint32_t)(p.NCS - 1);
  }
  __syncthreads();
  if (!sh_last) return;

  __threadfence();
  if (warp == 1) write_decision<false>(p, i, rs, decide_arrays(), rec.a, 0);  // the token at a comes last
  if (warp == 0) {
    // the partials of all chunks at once, one lane each
    const int lane = threadIdx.x & 31;
    KeyState all{INFINITY, INT_MAX};
    for (int k = lane; k < p.NCS; k += 32) {
      const RacePartial* src = p.race_part + (size_t)i * p.NCS + k;
      KeyState kr{__ldcg(&src->key_r), __ldcg(&src->idx_r)};
      if (key_better(kr, all)) all = kr;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      KeyState other{__shfl_xor_sync(0xFFFFFFFFu, all.key, o), __shfl_xor_sync(0xFFFFFFFFu, all.idx, o)};
      if (key_better(other, all)) all = other;
    }
    if (lane == 0) {
      p.counters[i] = 0u;  // leave the workspace zeroed for the next call
      sh_b = all.idx;
    }
  }
  __syncthreads();
  int b = sh_b;
  int wmode = mode;
  if (b == INT_MAX) {
    // Every weight is zero: an empty residual (p <= q in fp32, or p all on
    // the one-hot draft).  Draw from p instead, the whole row in this CTA.
    wmode = kWeightP;
    KeyState bp{INFINITY, INT_MAX};
    race_level1_any<T, kWeightP>(p, row, nullptr, 0, (V + kRaceQuad - 1) / kRaceQuad, warp, kSampleThreads / 32,
                                 ra, bp);
    bp = cta_min_key(bp, sh_red);
    if (threadIdx.x == 0) sh_b = bp.idx;
    __syncthreads();
    b = sh_b;
  }
  // ---- level 2 inside block b ----
  KeyState y{INFINITY, INT_MAX};
  if (b != INT_MAX) {
    if (wmode == kWeightResidual)
      y = race_level2<T, kWeightResidual>(row, qrow, p.q_dtype, V, 0, b, ra, sh_red);
    else if (wmode == kWeightExcl)
      y = race_level2<T, kWeightExcl>(row, qrow, p.q_dtype, V, 0, b, ra, sh_red);
    else
      y = race_level2<T, kWeightP>(row, qrow, p.q_dtype, V, 0, b, ra, sh_red);
  }
  if (threadIdx.x != 0) return;
  int32_t* tok = p.out_tokens + (size_t)i * (p.K + 1);
  if (y.idx == INT_MAX) {
    report(p.status, SPEC_ERR_BAD_INPUT);
    tok[rec.a] = -1;
    p.accepted_len[i] = 0;
    return;
  }
  tok[rec.a] = y.idx;
}

// ---------------------------------------------------------------------------
// Launcher
// ---------------------------------------------------------------------------
template <typename T>
static cudaError_t launch_typed(const VerifyLaunch& p, cudaStream_t stream, cudaEvent_t ev_before,
                                cudaEvent_t ev_after) {
  const bool greedy = p.temperature == 0.0f;
  const unsigned grid1 = (unsigned)((long long)p.B * (p.K + 1) * p.NC);
  if (ev_before) cudaEventRecord(ev_before, stream);
  cudaError_t err = greedy ? launch_after_previous(stream_rows_kernel<T, true>, dim3(grid1), dim3(kStreamThreads), 0,
                                                   stream, p)
                           : launch_after_previous(stream_rows_kernel<T, false>, dim3(grid1), dim3(kStreamThreads),
                                                   0, stream, p);
  if (err != cudaSuccess) return err;
  err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  if (ev_after) cudaEventRecord(ev_after, stream);
  if (greedy) {
    err = launch_after_previous(greedy_decide_kernel<T>, dim3((unsigned)p.B), dim3(32), 0, stream, p);
    if (err != cudaSuccess) return err;
    return cudaGetLastError();
  }
  // The sampling CTAs are launched while the streaming kernel drains and
  // wait (griddepcontrol.wait) for its completion.
  err = launch_after_previous(sample_kernel<T>, dim3((unsigned)((long long)p.B * p.NCS)), dim3(kSampleThreads), 0,
                              stream, p);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

cudaError_t launch_verify(const VerifyLaunch& p, cudaStream_t stream, cudaEvent_t ev_before,
                          cudaEvent_t ev_after) {
  if (p.logits_dtype == SPEC_F32) return launch_typed<float>(p, stream, ev_before, ev_after);
  return launch_typed<__nv_bfloat16>(p, stream, ev_before, ev_after);
}

}  // namespace spec
