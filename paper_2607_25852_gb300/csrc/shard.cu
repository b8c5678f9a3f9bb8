// shard.cu -- verification with the vocabulary split across tensor-parallel
// ranks (arxiv 2607.25852 serves its target with TP = 8, Section 4.4;
// Section 1 for the verification rule).
//
// Each rank holds the logits (and q) of a contiguous column range
// [v_begin, v_begin + V_shard) of the vocabulary, at any boundaries.  One
// round takes four calls and two small exchanges between them, which the
// caller makes (an all-gather of fixed-size records; on one GPU, records
// written side by side):
//
//   spec_shard_stats   (every rank)  per packed row: the shard's softmax
//                      statistics (max, sum) or (max, argmax), and the logit
//                      and q value at the row's draft if the shard owns the
//                      draft's column.  32-byte records [R_max].
//   -- all-gather of the S ranks' records --
//   spec_shard_decide  (every rank, identical results)  merges the S records
//                      per row in shard order, runs the decision chain and
//                      writes the committed prefix and, at t > 0, a 32-byte
//                      decision record per request.
//   spec_shard_sample  (every rank, t > 0)  level 1 of the two-level race over
//                      the blocks the shard owns whole, and level 2 inside the
//                      best of them; for a block that straddles a shard
//                      boundary, the shard's part of its weight sum and the
//                      best entry of that part.  96 B per request.
//   -- all-gather of the S ranks' race records --
//   spec_shard_finish  (every rank, t > 0)  completes the straddling blocks
//                      (their weight sums added over shards, their block
//                      variates drawn) and takes the lowest key over all
//                      blocks: the sampled token.
//
// The block and entry variates are those of spec_verify (they depend on the
// vocabulary index only).  At t = 0 the result equals spec_verify's bit for
// bit; at t > 0 shard sums merge in another order than spec_verify's chunk
// sums, so results agree within the same tolerance as against the oracle.
#include <float.h>
#include <math.h>

#include <algorithm>

#include "verify_common.cuh"

namespace spec {

// Per (shard, packed row).
struct alignas(16) ShardStat {
  float m;        // max logit over the shard's columns
  float s;        // t > 0: sum of 2^(l*c2 - fl(m*c2)); t = 0: unused
  int32_t idx;    // t = 0: lowest vocabulary index of the max (INT_MAX: none)
  int32_t flags;  // bit0: NaN (or +inf at t > 0) seen
  float lz;       // the row's draft: its logit, if the shard owns the draft's column
  float qz;       // ... and q there (1 for one-hot q)
  int32_t owned;  // 1 if the draft's column is in the shard
  int32_t pad;
};
static_assert(sizeof(ShardStat) == SPEC_SHARD_STAT_BYTES, "shard record size");

// A race block that straddles a shard boundary: this shard's part of it.
// "r" is the draw's weights, "p" the fallback race over p (at a rejection).
struct alignas(16) ShardPart {
  int32_t blk;    // block index (INT_MAX: no such part)
  float w_r;      // sum of the part's weights
  float w_p;
  float ek_r;     // lowest entry key E'_v / w_v of the part (INFINITY: none)
  int32_t ey_r;   // its entry (INT_MAX: none)
  float ek_p;
  int32_t ey_p;
  int32_t pad;
};

// Per (shard, request).
struct alignas(16) ShardRace {
  float key_r;     // best block the shard owns whole: its key,
  int32_t blk_r;   // index (INT_MAX: none)
  int32_t y_r;     // and the entry drawn in it (-1: none)
  int32_t empty;   // 1: no positive draw weight anywhere in the shard
  float key_p;     // the same for the race over p, drawn in only when empty
  int32_t blk_p;
  int32_t y_p;
  int32_t pad;
  ShardPart part[2];  // the straddling blocks at the shard's start and end
};
static_assert(sizeof(ShardRace) == SPEC_SHARD_RACE_BYTES, "shard race record size");
static_assert(sizeof(ReqRec) == SPEC_SHARD_DECISION_BYTES, "decision record size");

struct ShardLaunch {
  const void* logits;  // [R_max, Vs] of the shard
  int logits_dtype;
  const int32_t* row_offsets;
  const int32_t* depth;
  const int32_t* drafts;
  const void* q;  // [B, K, Vs] of the shard, or null (one-hot)
  int q_dtype;
  bool dense_q;
  int B, K, V;      // V: the whole vocabulary
  int v_begin, Vs;  // the shard's columns
  float temperature, c2, inv_t;
  const uint64_t* seeds;
  const uint64_t* request_ids;
  const int64_t* pos_base;
  int32_t* accepted_len;
  int32_t* out_tokens;
  float* p_draft;
  float* row_stats;
  int32_t* status;
  int R_max;
  int S;             // decide / finish: number of shards
  ShardStat* stats;  // stats: out [R_max]; decide: in [S][R_max]
  ReqRec* req_rec;   // decide: out [B]; sample / finish: in [B]
  ShardRace* races;  // sample: out [B]; finish: in [S][B]
  // workspace of stats / sample
  RowPartial* row_part;    // [R_max * NC]
  RacePartial* race_part;  // [B * NCS]
  ShardPart* part_ws;      // [B][2] the cut blocks' parts (sample)
  uint32_t* row_count;     // [R_max] arrivals per row (stats)
  uint32_t* req_count;     // [B] arrivals per request (sample)
  int NC, chunk;           // stats: chunks per row and their length
  int NCS, quads_s, q0;    // sample: chunks, quads per chunk, first quad
  bool vec_s;
};

struct ShardGeometry {
  int NC, chunk;  // streaming pass over V_shard columns
  int quads_s;    // race quads per sampling chunk
  int NCS_max;    // sampling chunks for any shard start
  size_t row_part_off, race_part_off, part_off, counters_off, bytes;
};

static inline size_t round256(size_t x) { return (x + 255) / 256 * 256; }

static ShardGeometry shard_geometry(int B, int K, int Vs) {
  const VerifyGeometry g = verify_geometry(B, K, Vs);
  ShardGeometry s;
  // Streaming pass: aim for ~4096 (row, chunk) CTAs, each a whole number of
  // load rounds (256 threads x 8 16-byte vectors = 16384 bf16 entries), so
  // that only the last chunk of a row ends in a partial round.
  const long long R = (long long)B * (K + 1);
  long long nc = (4096 + R - 1) / R;
  nc = std::max(1LL, std::min(nc, std::max(1LL, (long long)Vs / 16384)));
  const long long chunk = ((Vs + nc - 1) / nc + 16383) / 16384 * 16384;
  s.NC = (int)((Vs + chunk - 1) / chunk);  // every chunk non-empty
  s.chunk = (int)chunk;
  s.quads_s = g.chunk_s / kRaceQuad;
  // a shard of Vs columns spans at most ceil(Vs / 1024) + 1 quads
  const long long nq_max = (Vs + kRaceQuad - 1) / kRaceQuad + 1;
  s.NCS_max = (int)((nq_max + s.quads_s - 1) / s.quads_s);
  const size_t R_max = (size_t)B * (K + 1);
  s.row_part_off = 0;
  s.race_part_off = round256(sizeof(RowPartial) * R_max * s.NC);
  s.part_off = s.race_part_off + round256(sizeof(RacePartial) * (size_t)B * s.NCS_max);
  s.counters_off = s.part_off + round256(sizeof(ShardPart) * 2 * (size_t)B);
  s.bytes = s.counters_off + round256(sizeof(uint32_t) * (R_max + (size_t)B));
  return s;
}

// ---------------------------------------------------------------------------
// spec_shard_stats: one CTA per (request, row, chunk of the shard); the last
// CTA of a row to finish merges the row's chunk partials into its record.
// ---------------------------------------------------------------------------
// The row's draft, seen from this shard: its logit and q value if the shard
// owns the draft's column.  The draft token is loaded before the stream, the
// logit and q value after it (no dependent round trips ahead of the loads).
struct DraftView {
  float lz, qz;
  int32_t owned;
};
template <typename T>
__device__ __forceinline__ DraftView draft_view(const ShardLaunch& p, int i, int j, int z, const T* row) {
  DraftView d{0.0f, 1.0f, 0};
  if (z >= p.v_begin && z < p.v_begin + p.Vs) {
    d.owned = 1;
    d.lz = load_elem(row + (z - p.v_begin));
    if (p.dense_q) d.qz = load_any(p.q, p.q_dtype, ((int64_t)i * p.K + j) * (int64_t)p.Vs + (z - p.v_begin));
  }
  return d;
}

__device__ __forceinline__ void write_stat(const ShardLaunch& p, long long r, float m, float s, int32_t idx,
                                           int32_t flags, const DraftView& d) {
  ShardStat st;
  st.m = m;
  st.s = s;
  st.idx = idx;
  st.flags = flags;
  st.lz = d.lz;
  st.qz = d.qz;
  st.owned = d.owned;
  st.pad = 0;
  p.stats[r] = st;
}

// kThreads = 256 (four CTAs per SM) or 128 (eight per SM): the same threads
// and loads in flight per SM either way.
template <typename T, bool kGreedy, int kThreads>
__global__ void __launch_bounds__(kThreads, 1024 / kThreads) shard_stats_kernel(const ShardLaunch p) {
  const int per_req = (p.K + 1) * p.NC;
  const int i = blockIdx.x / per_req;
  const int rem = blockIdx.x - i * per_req;
  const int j = rem / p.NC;
  const int c = rem - j * p.NC;
  pdl_wait_prerequisites();
  const ReqShape rs = request_shape(p, i);
  if (!rs.valid || j > rs.n) return;  // spec_shard_decide reports invalid requests
  pdl_launch_dependents();
  const long long r = rs.row0 + j;
  const T* row = static_cast<const T*>(p.logits) + (size_t)r * (size_t)p.Vs;
  // the row's draft (thread 0; -1 past the request's depth)
  const int z = threadIdx.x == 0 && j < rs.n ? __ldg(p.drafts + (size_t)i * p.K + j) : -1;
  RowAcc<T, kGreedy> acc;
  const int v0 = c * p.chunk;
  stream_chunk<T, kGreedy, kThreads, kUnroll, true>(acc, row, v0, min(p.Vs, v0 + p.chunk), p.v_begin, p.c2);
  DraftView dv{0.0f, 1.0f, 0};
  if (threadIdx.x == 0) dv = draft_view(p, i, j, z, row);
  const RowPartial part = cta_reduce_partial<T, kGreedy, kThreads>(acc, p.c2);
  if (p.NC == 1) {  // the whole shard row in this CTA: its partial is the record
    if (threadIdx.x == 0) write_stat(p, r, part.m, part.s, kGreedy ? part.idx : INT_MAX, part.flags, dv);
    return;
  }
  __shared__ int sh_last;
  if (threadIdx.x == 0) {
    p.row_part[(size_t)r * p.NC + c] = part;
    __threadfence();  // the partial before the count
    sh_last = atomicAdd(p.row_count + r, 1u) == (uint32_t)p.NC - 1u;
  }
  __syncthreads();
  if (!sh_last || threadIdx.x >= 32) return;
  __threadfence();  // the other CTAs' partials after their counts
  // warp 0: merge the row's chunk partials (lanes over chunks)
  const int lane = threadIdx.x;
  const RowPartial* rp = p.row_part + (size_t)r * p.NC;
  ShardStat st{};
  int32_t f = 0;
  if (kGreedy) {
    ArgState best{-INFINITY, INT_MAX};
    for (int cc = lane; cc < p.NC; cc += 32) {
      const RowPartial x = load_partial_cg(rp + cc);
      f |= x.flags;
      ArgState o{x.m, x.idx};
      if (arg_better(o, best)) best = o;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      ArgState other{__shfl_xor_sync(0xFFFFFFFFu, best.v, o), __shfl_xor_sync(0xFFFFFFFFu, best.idx, o)};
      if (arg_better(other, best)) best = other;
    }
    st.m = best.v;
    st.idx = best.idx;
  } else {
    SoftState all{-INFINITY, 0.0f};
    for (int cc = lane; cc < p.NC; cc += 32) {
      const RowPartial x = load_partial_cg(rp + cc);
      f |= x.flags;
      all = soft_merge(all, SoftState{x.m, x.s}, p.c2);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      SoftState other{__shfl_xor_sync(0xFFFFFFFFu, all.m, o), __shfl_xor_sync(0xFFFFFFFFu, all.s, o)};
      all = soft_merge(all, other, p.c2);
    }
    st.m = all.m;
    st.s = all.s;
    st.idx = INT_MAX;
  }
  st.flags = (int32_t)__reduce_or_sync(0xFFFFFFFFu, (unsigned)f);
  if (lane == 0) {
    write_stat(p, r, st.m, st.s, st.idx, st.flags, dv);
    p.row_count[r] = 0u;  // leave the workspace zeroed for the next call
  }
}

template <typename T, bool kGreedy>
static cudaError_t launch_stats(unsigned grid, bool narrow, cudaStream_t stream, const ShardLaunch& p) {
  return narrow ? launch_after_previous(shard_stats_kernel<T, kGreedy, 128>, dim3(grid), dim3(128), 0, stream, p)
                : launch_after_previous(shard_stats_kernel<T, kGreedy, 256>, dim3(grid), dim3(256), 0, stream, p);
}

// ---------------------------------------------------------------------------
// spec_shard_decide: one warp per request.
// ---------------------------------------------------------------------------
template <bool kGreedy>
__global__ void __launch_bounds__(32) shard_decide_kernel(const ShardLaunch p) {
  const int i = blockIdx.x;
  const int lane = threadIdx.x;
  pdl_wait_prerequisites();
  __shared__ float sh_m[kMaxRows];
  __shared__ float sh_S[kMaxRows];
  __shared__ int32_t sh_g[kMaxRows];
  __shared__ int32_t sh_z[kMaxRows];
  __shared__ float sh_pz[kMaxRows];
  __shared__ float sh_lq[kMaxRows];
  const ReqShape rs = request_shape(p, i);
  const DecidePre pre = decide_prefetch<ShardLaunch, false, !kGreedy>(p, i);
  const int n = rs.n;
  const long long row0 = rs.row0;
#pragma unroll
  for (int u = 0; u < (kMaxRows + 31) / 32; ++u)
    if (lane + 32 * u < p.K) sh_z[lane + 32 * u] = pre.z[u];
  __syncwarp();
  int bad = rs.valid ? 0 : 1;
  float lz[(kMaxRows + 31) / 32], qz[(kMaxRows + 31) / 32];
#pragma unroll
  for (int u = 0; u < (kMaxRows + 31) / 32; ++u) {
    lz[u] = 0.0f;
    qz[u] = 1.0f;
  }
  if (rs.valid) {
    // rows (a lane per row): the S shard records merged in shard order, their
    // loads issued kBatch at a time; the draft fields come with them
    constexpr int kBatch = 8;
    const uint4* rec = reinterpret_cast<const uint4*>(p.stats);
    for (int j = lane; j <= n; j += 32) {
      int32_t f = 0;
      ArgState best{-INFINITY, INT_MAX};
      SoftState all{-INFINITY, 0.0f};
      int owners = 0;
      float lzj = 0.0f, qzj = 1.0f;
      for (int s0 = 0; s0 < p.S; s0 += kBatch) {
        uint4 a[kBatch], b[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          if (s0 + u < p.S) {
            const size_t k = 2 * ((size_t)(s0 + u) * p.R_max + row0 + j);
            a[u] = rec[k];
            if (j < n) b[u] = rec[k + 1];
          }
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          if (s0 + u >= p.S) break;
          f |= (int32_t)a[u].w;
          if (kGreedy) {
            const ArgState o{__uint_as_float(a[u].x), (int32_t)a[u].z};
            if (arg_better(o, best)) best = o;
          } else {
            all = soft_merge(all, SoftState{__uint_as_float(a[u].x), __uint_as_float(a[u].y)}, p.c2);
          }
          if (j < n && b[u].z) {
            ++owners;
            lzj = __uint_as_float(b[u].x);
            qzj = __uint_as_float(b[u].y);
          }
        }
      }
      if (kGreedy) {
        sh_m[j] = best.v;
        sh_g[j] = best.idx;
        if (f || best.idx == INT_MAX) bad = 1;
      } else {
        sh_m[j] = all.m;
        sh_S[j] = all.s;
        sh_pz[j] = lzj;  // staged here; decide_chain overwrites it with p(z)
        sh_lq[j] = qzj;
        if (f || !(all.m > -INFINITY) || !(all.s > 0.0f) || !isfinite(all.s)) bad = 1;
      }
      // the shards must cover the draft's column exactly once
      if (j < n && (owners != 1 || sh_z[j] < 0 || sh_z[j] >= p.V)) bad = 1;
    }
    if (!kGreedy) {
      __syncwarp();
#pragma unroll
      for (int u = 0; u < (kMaxRows + 31) / 32; ++u) {
        const int j = lane + 32 * u;
        if (j < n) {
          lz[u] = sh_pz[j];
          qz[u] = sh_lq[j];
        }
      }
    }
  }
  bad = __any_sync(0xFFFFFFFFu, bad);
  __syncwarp();
  decide_chain<kGreedy>(p, i, rs, pre, DecideArrays{sh_m, sh_S, sh_g, sh_z, sh_pz}, lz, qz, bad, true, p.req_rec + i);
}

// ---------------------------------------------------------------------------
// spec_shard_sample: one CTA per (request, chunk of the shard's quads).
// ---------------------------------------------------------------------------
// Level 1 over quads [q_first, q_end), blocks the shard owns whole.  At a
// rejection (kDual) the race over p runs beside it on the same variates: if no
// shard has a positive draw weight, the draw falls back to p, as in
// spec_verify.
template <typename T, int kMode, bool kDual>
__device__ __forceinline__ void shard_level1(const ShardLaunch& p, const T* row, const void* qrow, int q_first,
                                             int q_end, const RaceArgs& ra, KeyState& best, KeyState& best_p) {
  const int warp = threadIdx.x >> 5;
  const int vend = p.v_begin + p.Vs;
  const bool tail_whole = vend == p.V;
  constexpr int kW = kSampleThreads / 32;
  if (p.vec_s) {
    if (kMode == kWeightResidual && p.q_dtype == SPEC_F32)
      race_level1_impl<T, float, kMode, kSrcGlobalVec, kDual, true>(row, qrow, p.q_dtype, vend, p.v_begin, q_first,
                                                                    q_end, warp, kW, ra, best, best_p, p.v_begin,
                                                                    tail_whole);
    else
      race_level1_impl<T, __nv_bfloat16, kMode, kSrcGlobalVec, kDual, true>(
          row, qrow, p.q_dtype, vend, p.v_begin, q_first, q_end, warp, kW, ra, best, best_p, p.v_begin, tail_whole);
  } else {
    race_level1_impl<T, T, kMode, kSrcGlobalScalar, kDual, true>(row, qrow, p.q_dtype, vend, p.v_begin, q_first,
                                                                 q_end, warp, kW, ra, best, best_p, p.v_begin,
                                                                 tail_whole);
  }
}

template <typename T>
__device__ __forceinline__ KeyState shard_level2(const ShardLaunch& p, int mode, const T* row, const void* qrow, int b,
                                                 const RaceArgs& ra, KeyState* sh) {
  const int vend = p.v_begin + p.Vs;
  if (mode == kWeightResidual) return race_level2<T, kWeightResidual>(row, qrow, p.q_dtype, vend, p.v_begin, b, ra, sh);
  if (mode == kWeightExcl) return race_level2<T, kWeightExcl>(row, qrow, p.q_dtype, vend, p.v_begin, b, ra, sh);
  return race_level2<T, kWeightP>(row, qrow, p.q_dtype, vend, p.v_begin, b, ra, sh);
}

// The lowest keys a and b over the CTA in one exchange (results in thread 0;
// sh: 2 x kSampleThreads / 32 slots).
__device__ __forceinline__ void cta_min_key2(KeyState& a, KeyState& b, KeyState* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const KeyState oa{__shfl_xor_sync(0xFFFFFFFFu, a.key, o), __shfl_xor_sync(0xFFFFFFFFu, a.idx, o)};
    const KeyState ob{__shfl_xor_sync(0xFFFFFFFFu, b.key, o), __shfl_xor_sync(0xFFFFFFFFu, b.idx, o)};
    if (key_better(oa, a)) a = oa;
    if (key_better(ob, b)) b = ob;
  }
  if (lane == 0) {
    sh[warp] = a;
    sh[kSampleThreads / 32 + warp] = b;
  }
  __syncthreads();
  if (threadIdx.x == 0)
    for (int k = 0; k < kSampleThreads / 32; ++k) {
      if (key_better(sh[k], a)) a = sh[k];
      if (key_better(sh[kSampleThreads / 32 + k], b)) b = sh[kSampleThreads / 32 + k];
    }
  __syncthreads();
}

// The shard's part [lo, hi) of block b (one entry per thread): the part's
// weight sums (a warp butterfly, then the warps' sums in warp order) and
// lowest entry keys, from one exchange over the CTA.  Result in thread 0.
template <typename T>
__device__ ShardPart shard_part(const ShardLaunch& p, int mode, const T* row, const void* qrow, int b, int lo, int hi,
                                const RaceArgs& ra, KeyState* sh_key, float* sh_f) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int v = b * kRaceBlock + (int)threadIdx.x;
  float w = 0.0f, wp = 0.0f;
  KeyState er{INFINITY, INT_MAX}, ep{INFINITY, INT_MAX};
  if (v >= lo && v < hi) {
    const float x = load_elem(row + (v - p.v_begin));
    const float qv = mode == kWeightResidual ? load_any(qrow, p.q_dtype, v - p.v_begin) : 0.0f;
    const float ew = p_weight(x, ra.c2, ra.M2);
    w = mode == kWeightResidual ? weight_of<kWeightResidual>(ew, qv, v, ra.invS, ra.z_excl)
        : mode == kWeightExcl   ? weight_of<kWeightExcl>(ew, qv, v, ra.invS, ra.z_excl)
                                : ew;
    wp = mode == kWeightP ? 0.0f : ew;
    const uint4 r = philox(draw_counter(ra.position, ra.req, SPEC_PURPOSE_SAMPLE_IN_BLOCK, (uint32_t)(v >> 2)), ra.k0,
                           ra.k1);
    const uint32_t m = race_m((v & 3) == 0 ? r.x : (v & 3) == 1 ? r.y : (v & 3) == 2 ? r.z : r.w);
    if (w > 0.0f) er = KeyState{race_key(m, w), v};
    if (wp > 0.0f) ep = KeyState{race_key(m, wp), v};
  }
  ShardPart out;
  out.blk = b;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    w += __shfl_xor_sync(0xFFFFFFFFu, w, o);
    wp += __shfl_xor_sync(0xFFFFFFFFu, wp, o);
  }
  if (lane == 0) {
    sh_f[warp] = w;
    sh_f[kSampleThreads / 32 + warp] = wp;
  }
  cta_min_key2(er, ep, sh_key);  // its barriers also publish sh_f
  float t = 0.0f, tp = 0.0f;
#pragma unroll
  for (int k = 0; k < kSampleThreads / 32; ++k) {
    t += sh_f[k];
    tp += sh_f[kSampleThreads / 32 + k];
  }
  __syncthreads();  // sh_f is reused by the next part
  out.w_r = t;
  out.w_p = tp;
  out.ek_r = er.key;
  out.ey_r = er.idx;
  out.ek_p = ep.key;
  out.ey_p = ep.idx;
  out.pad = 0;
  return out;
}

// A part written by another CTA of this grid: read at L2 (.cg).
__device__ __forceinline__ ShardPart load_part_cg(const ShardPart* ptr) {
  const uint4 a = __ldcg(reinterpret_cast<const uint4*>(ptr));
  const uint4 b = __ldcg(reinterpret_cast<const uint4*>(ptr) + 1);
  ShardPart x;
  x.blk = (int32_t)a.x;
  x.w_r = __uint_as_float(a.y);
  x.w_p = __uint_as_float(a.z);
  x.ek_r = __uint_as_float(a.w);
  x.ey_r = (int32_t)b.x;
  x.ek_p = __uint_as_float(b.y);
  x.ey_p = (int32_t)b.z;
  x.pad = (int32_t)b.w;
  return x;
}

__device__ __forceinline__ ShardPart no_part() {
  ShardPart n;
  n.blk = INT_MAX;
  n.w_r = n.w_p = 0.0f;
  n.ek_r = n.ek_p = INFINITY;
  n.ey_r = n.ey_p = INT_MAX;
  n.pad = 0;
  return n;
}

template <typename T>
__global__ void __launch_bounds__(kSampleThreads, 4) shard_sample_kernel(const ShardLaunch p) {
  __shared__ int sh_last, sh_b, sh_bp;
  __shared__ float sh_kb, sh_kbp;
  __shared__ KeyState sh_red[2 * (kSampleThreads / 32)];
  __shared__ float sh_f[2 * (kSampleThreads / 32)];
  const int i = blockIdx.x / p.NCS;
  const int cs = blockIdx.x - i * p.NCS;
  pdl_wait_prerequisites();
  pdl_launch_dependents();
  const ReqRec rec = p.req_rec[i];
  if (rec.flags & 1) return;  // bad input: the decision wrote the outputs
  if (rec.a < 0 || rec.a > p.K || rec.srow < 0 || rec.srow >= p.R_max || rec.z_excl < -1 || rec.z_excl >= p.V ||
      ((rec.flags & 4) && (!p.dense_q || rec.a >= p.K))) {
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
  const int mode = (rec.flags & 4) ? kWeightResidual : (rec.flags & 2) ? kWeightExcl : kWeightP;
  const T* row = static_cast<const T*>(p.logits) + (size_t)rec.srow * p.Vs;
  const size_t qsize = p.q_dtype == SPEC_F32 ? 4 : 2;
  const void* qrow = mode == kWeightResidual
                         ? (const void*)((const char*)p.q + ((size_t)i * p.K + rec.a) * (size_t)p.Vs * qsize)
                         : nullptr;
  const int vend = p.v_begin + p.Vs;
  // ---- level 1 over this CTA's quads ----
  const int q_first = p.q0 + cs * p.quads_s;
  const int q_end = min((vend + kRaceQuad - 1) / kRaceQuad, q_first + p.quads_s);
  KeyState best{INFINITY, INT_MAX}, best_p{INFINITY, INT_MAX};
  if (mode == kWeightResidual)
    shard_level1<T, kWeightResidual, true>(p, row, qrow, q_first, q_end, ra, best, best_p);
  else if (mode == kWeightExcl)
    shard_level1<T, kWeightExcl, true>(p, row, qrow, q_first, q_end, ra, best, best_p);
  else
    shard_level1<T, kWeightP, false>(p, row, qrow, q_first, q_end, ra, best, best_p);
  cta_min_key2(best, best_p, sh_red);
  // ---- the cut blocks at the shard's ends: the first and the last chunk's
  // CTA compute the shard's part of each before arriving ----
  const int hb = p.v_begin / kRaceBlock;   // block holding the first column
  const int tb = (vend - 1) / kRaceBlock;  // block holding the last column
  const bool head_part = p.v_begin % kRaceBlock != 0 || (vend < p.V && vend % kRaceBlock != 0 && tb == hb);
  const bool tail_part = vend < p.V && vend % kRaceBlock != 0 && tb != hb;
  if (cs == 0 && head_part) {
    const ShardPart pt = shard_part<T>(p, mode, row, qrow, hb, p.v_begin, tb == hb ? vend : (hb + 1) * kRaceBlock,
                                       ra, sh_red, sh_f);
    if (threadIdx.x == 0) p.part_ws[2 * (size_t)i] = pt;
  }
  if (cs == p.NCS - 1 && tail_part) {
    const ShardPart pt = shard_part<T>(p, mode, row, qrow, tb, tb * kRaceBlock, vend, ra, sh_red, sh_f);
    if (threadIdx.x == 0) p.part_ws[2 * (size_t)i + 1] = pt;
  }
  if (threadIdx.x == 0) {
    RacePartial rp;
    rp.key_r = best.key;
    rp.idx_r = best.idx;
    rp.key_p = best_p.key;
    rp.idx_p = best_p.idx;
    p.race_part[(size_t)i * p.NCS + cs] = rp;
    __threadfence();
    sh_last = atomicAdd(p.req_count + i, 1u) == (uint32_t)(p.NCS - 1);
  }
  __syncthreads();
  if (!sh_last) return;
  __threadfence();
  // ---- the last CTA of the request: merge the chunks' bests ----
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    KeyState r{INFINITY, INT_MAX}, q{INFINITY, INT_MAX};
    for (int k = lane; k < p.NCS; k += 32) {
      const uint4 w = __ldcg(reinterpret_cast<const uint4*>(p.race_part + (size_t)i * p.NCS + k));
      const KeyState kr{__uint_as_float(w.x), (int32_t)w.y}, kp{__uint_as_float(w.z), (int32_t)w.w};
      if (key_better(kr, r)) r = kr;
      if (key_better(kp, q)) q = kp;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const KeyState orr{__shfl_xor_sync(0xFFFFFFFFu, r.key, o), __shfl_xor_sync(0xFFFFFFFFu, r.idx, o)};
      const KeyState oq{__shfl_xor_sync(0xFFFFFFFFu, q.key, o), __shfl_xor_sync(0xFFFFFFFFu, q.idx, o)};
      if (key_better(orr, r)) r = orr;
      if (key_better(oq, q)) q = oq;
    }
    if (lane == 0) {
      p.req_count[i] = 0u;  // leave the workspace zeroed for the next call
      sh_b = r.idx;
      sh_kb = r.key;
      sh_bp = q.idx;
      sh_kbp = q.key;
    }
  }
  __syncthreads();
  const int b = sh_b, bp = sh_bp;
  ShardPart part[2] = {no_part(), no_part()};
  if (head_part) part[0] = load_part_cg(p.part_ws + 2 * (size_t)i);
  if (tail_part) part[1] = load_part_cg(p.part_ws + 2 * (size_t)i + 1);
  const bool empty = b == INT_MAX && !(part[0].w_r > 0.0f) && !(part[1].w_r > 0.0f);
  // ---- level 2 in the best whole block ----
  ShardRace out;
  out.key_r = sh_kb;
  out.blk_r = b;
  out.y_r = -1;
  out.empty = empty ? 1 : 0;
  out.key_p = INFINITY;
  out.blk_p = INT_MAX;
  out.y_p = -1;
  out.pad = 0;
  if (b != INT_MAX) {
    const KeyState y = shard_level2<T>(p, mode, row, qrow, b, ra, sh_red);
    out.y_r = y.idx == INT_MAX ? -1 : y.idx;
  } else if (mode != kWeightP && empty && bp != INT_MAX) {
    // no positive draw weight in this shard: its whole-block part of the
    // fallback race over p
    const KeyState y = shard_level2<T>(p, kWeightP, row, nullptr, bp, ra, sh_red);
    out.key_p = sh_kbp;
    out.blk_p = bp;
    out.y_p = y.idx == INT_MAX ? -1 : y.idx;
  }
  out.part[0] = part[0];
  out.part[1] = part[1];
  if (threadIdx.x == 0) p.races[i] = out;
}

// ---------------------------------------------------------------------------
// spec_shard_finish: one warp per request.
// ---------------------------------------------------------------------------
// The level-1 race word of block b.
__device__ __forceinline__ uint32_t block_word(int b, const RaceArgs& a) {
  const uint4 r = philox(draw_counter(a.position, a.req, SPEC_PURPOSE_SAMPLE, (uint32_t)(b >> 2)), a.k0, a.k1);
  return (b & 3) == 0 ? r.x : (b & 3) == 1 ? r.y : (b & 3) == 2 ? r.z : r.w;
}

// Candidate block b with weight sum W (summed over its parts) and race word
// `word`: key E_b / W.
__device__ __forceinline__ void finish_block(KeyState& best, int& y, int b, float W, int y_part, uint32_t word) {
  if (!(W > 0.0f)) return;
  const KeyState k{race_key(race_m(word), W), b};
  if (key_better(k, best)) {
    best = k;
    y = y_part;
  }
}

// One warp per request: the lanes load up to 32 shards' records at a time
// into shared memory, lane 0 merges them in shard order.
constexpr int kFinishWarps = 4;

__global__ void __launch_bounds__(32 * kFinishWarps) shard_finish_kernel(const ShardLaunch p) {
  __shared__ ShardRace sh_rec[kFinishWarps][32];
  __shared__ uint32_t sh_word[kFinishWarps][32][2];  // the race words of the records' cut blocks
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * kFinishWarps + warp;
  pdl_wait_prerequisites();
  if (i >= p.B) return;
  const ReqRec rec = p.req_rec[i];
  if (rec.flags & 1) return;
  if (rec.a < 0 || rec.a > p.K) {
    if (lane == 0) report(p.status, SPEC_ERR_WORKSPACE);
    return;
  }
  RaceArgs a{};
  a.position = rec.position;
  a.req = __ldg(reinterpret_cast<const unsigned long long*>(p.request_ids) + i);
  const uint64_t seed = __ldg(reinterpret_cast<const unsigned long long*>(p.seeds) + i);
  a.k0 = (uint32_t)seed;
  a.k1 = (uint32_t)(seed >> 32);
  KeyState r{INFINITY, INT_MAX}, q{INFINITY, INT_MAX};
  int yr = -1, yq = -1;
  // cut blocks: the parts of one block are adjacent in shard order
  int cur = INT_MAX;
  uint32_t cur_word = 0;
  float Wr = 0.0f, Wp = 0.0f;
  KeyState er{INFINITY, INT_MAX}, ep{INFINITY, INT_MAX};
  for (int s0 = 0; s0 < p.S; s0 += 32) {
    __syncwarp();
    if (s0 + lane < p.S) {
      const uint4* src = reinterpret_cast<const uint4*>(p.races + (size_t)(s0 + lane) * p.B + i);
      uint4* dst = reinterpret_cast<uint4*>(&sh_rec[warp][lane]);
#pragma unroll
      for (int w = 0; w < (int)(sizeof(ShardRace) / 16); ++w) dst[w] = src[w];
      // the race words of this record's cut blocks, a lane per record (lane
      // 0 then merges the records in shard order)
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int b = sh_rec[warp][lane].part[h].blk;
        sh_word[warp][lane][h] = b != INT_MAX ? block_word(b, a) : 0u;
      }
    }
    __syncwarp();
    if (lane != 0) continue;
    for (int s = s0; s < min(p.S, s0 + 32); ++s) {
      const ShardRace& x = sh_rec[warp][s - s0];
      const KeyState kr{x.key_r, x.blk_r}, kp{x.key_p, x.blk_p};
      if (x.blk_r != INT_MAX && key_better(kr, r)) {
        r = kr;
        yr = x.y_r;
      }
      if (x.blk_p != INT_MAX && key_better(kp, q)) {
        q = kp;
        yq = x.y_p;
      }
      for (int h = 0; h < 2; ++h) {
        const ShardPart& pt = x.part[h];
        if (pt.blk == INT_MAX) continue;
        if (pt.blk != cur) {
          if (cur != INT_MAX) {
            finish_block(r, yr, cur, Wr, er.idx, cur_word);
            finish_block(q, yq, cur, Wp, ep.idx, cur_word);
          }
          cur = pt.blk;
          cur_word = sh_word[warp][s - s0][h];
          Wr = Wp = 0.0f;
          er = ep = KeyState{INFINITY, INT_MAX};
        }
        Wr += pt.w_r;
        Wp += pt.w_p;
        const KeyState kr2{pt.ek_r, pt.ey_r}, kp2{pt.ek_p, pt.ey_p};
        if (pt.ey_r != INT_MAX && key_better(kr2, er)) er = kr2;
        if (pt.ey_p != INT_MAX && key_better(kp2, ep)) ep = kp2;
      }
    }
  }
  if (lane != 0) return;
  if (cur != INT_MAX) {
    finish_block(r, yr, cur, Wr, er.idx, cur_word);
    finish_block(q, yq, cur, Wp, ep.idx, cur_word);
  }
  const int y = r.idx != INT_MAX ? yr : yq;
  int32_t* tok = p.out_tokens + (size_t)i * (p.K + 1);
  if (y < 0 || y >= p.V) {
    report(p.status, SPEC_ERR_BAD_INPUT);
    tok[rec.a] = -1;
    p.accepted_len[i] = 0;
    return;
  }
  tok[rec.a] = y;
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
static bool shard_shape_ok(int B, int K, int V, int v_begin, int Vs) {
  return B >= 1 && K >= 0 && K <= SPEC_MAX_DRAFTS && V >= 1 && V < SPEC_MAX_VOCAB && Vs >= 1 && v_begin >= 0 &&
         (long long)v_begin + Vs <= V && (long long)B * (K + 1) <= (1LL << 28);
}

static void fill_common(ShardLaunch& p, int B, int K, int V, float temperature) {
  p.B = B;
  p.K = K;
  p.V = V;
  p.temperature = temperature;
  p.c2 = temperature > 0.0f ? (float)(1.4426950408889634 / (double)temperature) : 0.0f;
  p.inv_t = temperature > 0.0f ? (float)(1.0 / (double)temperature) : 0.0f;
  p.R_max = B * (K + 1);
}

static bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

}  // namespace spec

using spec::ShardLaunch;

extern "C" size_t spec_shard_workspace(int B, int K, int V_shard) {
  if (B < 1 || K < 0 || K > SPEC_MAX_DRAFTS || V_shard < 1 || V_shard >= SPEC_MAX_VOCAB ||
      (long long)B * (K + 1) > (1LL << 28))
    return 0;
  return spec::shard_geometry(B, K, V_shard).bytes;
}

extern "C" int spec_shard_stats(const void* logits_shard, int logits_dtype, const int32_t* row_offsets,
                                const int32_t* depth, const int32_t* draft_tokens, const void* q_shard, int q_dtype,
                                int B, int K, int V, int v_begin, int V_shard, float temperature,
                                const int64_t* pos_base, void* stats_out, int32_t* status, void* ws,
                                size_t ws_bytes, cudaStream_t stream) {
  spec::NvtxRange range("spec_shard_stats");
  if (!spec::shard_shape_ok(B, K, V, v_begin, V_shard)) return SPEC_ERR_INVALID_ARG;
  if ((logits_dtype != SPEC_BF16 && logits_dtype != SPEC_F32) || !(temperature >= 0.0f) || isinf(temperature))
    return SPEC_ERR_INVALID_ARG;
  if (q_shard && q_dtype != SPEC_BF16 && q_dtype != SPEC_F32) return SPEC_ERR_INVALID_ARG;
  if (!logits_shard || (K > 0 && !draft_tokens) || !pos_base || !stats_out) return SPEC_ERR_INVALID_ARG;
  const spec::ShardGeometry g = spec::shard_geometry(B, K, V_shard);
  if (!ws || ws_bytes < g.bytes || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return SPEC_ERR_WORKSPACE;
  if (!spec::aligned16(stats_out)) return SPEC_ERR_INVALID_ARG;
  ShardLaunch p{};
  spec::fill_common(p, B, K, V, temperature);
  p.logits = logits_shard;
  p.logits_dtype = logits_dtype;
  p.row_offsets = row_offsets;
  p.depth = depth;
  p.drafts = draft_tokens;
  p.q = temperature > 0.0f ? q_shard : nullptr;
  p.q_dtype = q_dtype;
  p.dense_q = p.q != nullptr;
  p.v_begin = v_begin;
  p.Vs = V_shard;
  p.pos_base = pos_base;
  p.status = status;
  p.stats = static_cast<spec::ShardStat*>(stats_out);
  char* base = static_cast<char*>(ws);
  p.row_part = reinterpret_cast<spec::RowPartial*>(base + g.row_part_off);
  p.row_count = reinterpret_cast<uint32_t*>(base + g.counters_off);
  p.NC = g.NC;
  p.chunk = g.chunk;
  const unsigned grid = (unsigned)((long long)B * (K + 1) * p.NC);
  // 256-thread CTAs while the grid fits in one wave of them (four per SM),
  // else 128-thread CTAs (eight per SM), which take twice the rows into the
  // first wave
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return SPEC_ERR_CUDA;
  const bool narrow = (long long)grid > 4LL * sms;
  const bool greedy = temperature == 0.0f;
  cudaError_t err;
  if (logits_dtype == SPEC_F32)
    err = greedy ? spec::launch_stats<float, true>(grid, narrow, stream, p)
                 : spec::launch_stats<float, false>(grid, narrow, stream, p);
  else
    err = greedy ? spec::launch_stats<__nv_bfloat16, true>(grid, narrow, stream, p)
                 : spec::launch_stats<__nv_bfloat16, false>(grid, narrow, stream, p);
  if (err != cudaSuccess || cudaGetLastError() != cudaSuccess) return SPEC_ERR_CUDA;
  return SPEC_OK;
}

extern "C" int spec_shard_decide(const void* stats, int S, const int32_t* row_offsets, const int32_t* depth,
                                 const int32_t* draft_tokens, int q_dense, int B, int K, int V, float temperature,
                                 const uint64_t* seeds, const uint64_t* request_ids, const int64_t* pos_base,
                                 int32_t* accepted_len_out, int32_t* out_tokens, float* p_draft_out,
                                 float* row_stats_out, void* decisions_out, int32_t* status, cudaStream_t stream) {
  spec::NvtxRange range("spec_shard_decide");
  if (!spec::shard_shape_ok(B, K, V, 0, V) || S < 1 || S > V) return SPEC_ERR_INVALID_ARG;
  if (!(temperature >= 0.0f) || isinf(temperature)) return SPEC_ERR_INVALID_ARG;
  if (!stats || (K > 0 && !draft_tokens) || !seeds || !request_ids || !pos_base || !accepted_len_out ||
      !out_tokens || (temperature > 0.0f && !decisions_out))
    return SPEC_ERR_INVALID_ARG;
  if (!spec::aligned16(stats) || (decisions_out && !spec::aligned16(decisions_out)) ||
      (row_stats_out && (reinterpret_cast<uintptr_t>(row_stats_out) & 7u) != 0))
    return SPEC_ERR_INVALID_ARG;
  ShardLaunch p{};
  spec::fill_common(p, B, K, V, temperature);
  p.S = S;
  p.stats = static_cast<spec::ShardStat*>(const_cast<void*>(stats));
  p.row_offsets = row_offsets;
  p.depth = depth;
  p.drafts = draft_tokens;
  p.dense_q = temperature > 0.0f && q_dense != 0;
  p.seeds = seeds;
  p.request_ids = request_ids;
  p.pos_base = pos_base;
  p.accepted_len = accepted_len_out;
  p.out_tokens = out_tokens;
  p.p_draft = p_draft_out;
  p.row_stats = row_stats_out;
  p.req_rec = static_cast<spec::ReqRec*>(decisions_out);
  p.status = status;
  const cudaError_t err =
      temperature == 0.0f
          ? spec::launch_after_previous(spec::shard_decide_kernel<true>, dim3(B), dim3(32), 0, stream, p)
          : spec::launch_after_previous(spec::shard_decide_kernel<false>, dim3(B), dim3(32), 0, stream, p);
  if (err != cudaSuccess || cudaGetLastError() != cudaSuccess) return SPEC_ERR_CUDA;
  return SPEC_OK;
}

extern "C" int spec_shard_sample(const void* logits_shard, int logits_dtype, const void* q_shard, int q_dtype,
                                 const void* decisions, int B, int K, int V, int v_begin, int V_shard,
                                 float temperature, const uint64_t* seeds, const uint64_t* request_ids,
                                 void* race_out, int32_t* status, void* ws, size_t ws_bytes, cudaStream_t stream) {
  spec::NvtxRange range("spec_shard_sample");
  if (!spec::shard_shape_ok(B, K, V, v_begin, V_shard)) return SPEC_ERR_INVALID_ARG;
  if ((logits_dtype != SPEC_BF16 && logits_dtype != SPEC_F32) || !(temperature >= 0.0f) || isinf(temperature))
    return SPEC_ERR_INVALID_ARG;
  if (temperature == 0.0f) return SPEC_OK;  // the argmax token is already written
  if (q_shard && q_dtype != SPEC_BF16 && q_dtype != SPEC_F32) return SPEC_ERR_INVALID_ARG;
  if (!logits_shard || !decisions || !seeds || !request_ids || !race_out) return SPEC_ERR_INVALID_ARG;
  if (!spec::aligned16(decisions) || !spec::aligned16(race_out)) return SPEC_ERR_INVALID_ARG;
  const spec::ShardGeometry g = spec::shard_geometry(B, K, V_shard);
  if (!ws || ws_bytes < g.bytes || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return SPEC_ERR_WORKSPACE;
  ShardLaunch p{};
  spec::fill_common(p, B, K, V, temperature);
  p.logits = logits_shard;
  p.logits_dtype = logits_dtype;
  p.q = q_shard;
  p.q_dtype = q_dtype;
  p.dense_q = q_shard != nullptr;
  p.v_begin = v_begin;
  p.Vs = V_shard;
  p.seeds = seeds;
  p.request_ids = request_ids;
  p.req_rec = static_cast<spec::ReqRec*>(const_cast<void*>(decisions));
  p.races = static_cast<spec::ShardRace*>(race_out);
  p.status = status;
  char* base = static_cast<char*>(ws);
  p.race_part = reinterpret_cast<spec::RacePartial*>(base + g.race_part_off);
  p.part_ws = reinterpret_cast<spec::ShardPart*>(base + g.part_off);
  p.req_count = reinterpret_cast<uint32_t*>(base + g.counters_off) + (size_t)B * (K + 1);
  // the shard's quads, in chunks of quads_s
  p.q0 = v_begin / spec::kRaceQuad;
  const int q1 = (v_begin + V_shard + spec::kRaceQuad - 1) / spec::kRaceQuad;
  p.quads_s = g.quads_s;
  p.NCS = (q1 - p.q0 + g.quads_s - 1) / g.quads_s;
  if (p.NCS > g.NCS_max) return SPEC_ERR_WORKSPACE;  // cannot happen: NCS_max covers every start
  // 16-byte level-1 loads: 8-entry groups of the vocabulary start on 16-byte
  // boundaries of the shard's rows
  const size_t esize = logits_dtype == SPEC_F32 ? 4 : 2, qsize = q_dtype == SPEC_F32 ? 4 : 2;
  const bool q_ok = !q_shard || (spec::aligned16(q_shard) && (V_shard * qsize) % 16 == 0);
  p.vec_s = v_begin % 8 == 0 && V_shard % 8 == 0 && spec::aligned16(logits_shard) && (V_shard * esize) % 16 == 0 &&
            q_ok;
  const unsigned grid = (unsigned)((long long)B * p.NCS);
  const cudaError_t err =
      logits_dtype == SPEC_F32
          ? spec::launch_after_previous(spec::shard_sample_kernel<float>, dim3(grid), dim3(spec::kSampleThreads), 0,
                                        stream, p)
          : spec::launch_after_previous(spec::shard_sample_kernel<__nv_bfloat16>, dim3(grid),
                                        dim3(spec::kSampleThreads), 0, stream, p);
  if (err != cudaSuccess || cudaGetLastError() != cudaSuccess) return SPEC_ERR_CUDA;
  return SPEC_OK;
}

extern "C" int spec_shard_finish(const void* races, int S, const void* decisions, int B, int K, int V,
                                 float temperature, const uint64_t* seeds, const uint64_t* request_ids,
                                 int32_t* accepted_len_out, int32_t* out_tokens, int32_t* status,
                                 cudaStream_t stream) {
  spec::NvtxRange range("spec_shard_finish");
  if (!spec::shard_shape_ok(B, K, V, 0, V) || S < 1 || S > V) return SPEC_ERR_INVALID_ARG;
  if (!(temperature >= 0.0f) || isinf(temperature)) return SPEC_ERR_INVALID_ARG;
  if (temperature == 0.0f) return SPEC_OK;
  if (!races || !decisions || !seeds || !request_ids || !accepted_len_out || !out_tokens) return SPEC_ERR_INVALID_ARG;
  if (!spec::aligned16(races) || !spec::aligned16(decisions)) return SPEC_ERR_INVALID_ARG;
  ShardLaunch p{};
  spec::fill_common(p, B, K, V, temperature);
  p.S = S;
  p.races = static_cast<spec::ShardRace*>(const_cast<void*>(races));
  p.req_rec = static_cast<spec::ReqRec*>(const_cast<void*>(decisions));
  p.seeds = seeds;
  p.request_ids = request_ids;
  p.accepted_len = accepted_len_out;
  p.out_tokens = out_tokens;
  p.status = status;
  const cudaError_t err =
      spec::launch_after_previous(spec::shard_finish_kernel, dim3((B + spec::kFinishWarps - 1) / spec::kFinishWarps),
                                  dim3(32 * spec::kFinishWarps), 0, stream, p);
  if (err != cudaSuccess || cudaGetLastError() != cudaSuccess) return SPEC_ERR_CUDA;
  return SPEC_OK;
}
