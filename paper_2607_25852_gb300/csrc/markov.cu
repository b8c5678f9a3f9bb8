// markov.cu -- the Markov head's sequential draw on sm_103a (arxiv
// 2607.25852, Section 3.2, Eq. dspark-markov: each position's base logits
// U_k get the first-order bias b_k = W1[x_{k-1}] W2 of the previously drawn
// token, q_k = softmax(U_k + b_k); the block distribution factorises over the
// positions, Eq. ar-factorization).
//
// Per position k, for all B requests at once, the bias is the dense
// contraction E_k W2 with E_k = W1[x_{k-1}] ([B, r] x [r, V]): it runs on the
// 5th-generation tensor cores.
//
//   markov_bias_kernel  persistent, one CTA per SM.  Warp 0 loads by TMA the
//                       operand E_k (128 x r; with B <= 64 rows 64..127
//                       repeat rows 0..63, other rows past B are zero) once,
//                       and the CTA's tiles of W2^T (128 vocabulary rows x r,
//                       128-byte swizzle), double-buffered.  Warp 1 issues
//                       tcgen05.mma (M = 128, N = 128, K = 16, bf16 -> fp32)
//                       into four TMEM accumulators.  Eight epilogue warps
//                       (two per TMEM lane quarter, alternate tiles) read the
//                       accumulator rows (tcgen05.ld, one request per
//                       thread; with the repeated rows, one column half of
//                       each tile per quarter pair), add U_k, and per
//                       64-column sub-block write its max and sum; they also
//                       keep the row's softmax statistics (or its argmax at
//                       tau = 0): four partials per request and CTA.
//   markov_pick_kernel  one CTA per request: merges the partials; at tau > 0
//                       forms the level-1 key of every 256-entry race block
//                       from its four sub-blocks, recomputes the winning
//                       block's 256 logits and draws inside it (level 2);
//                       writes the draft, its confidence and the row
//                       statistics, and gathers W1 at the draft into E for
//                       the next position.
//
// Consecutive kernels overlap through programmatic dependent launch: each
// triggers its dependent at entry, and the bias kernel loads its first W2^T
// tiles before it waits for the previous position's pick.
//
// Every mbarrier wait is bounded (about a second): a wait that gives up sets
// SPEC_ERR_TIMEOUT, the kernel stops issuing work, waits (bounded) for what
// it issued, frees its TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>

#include "verify_common.cuh"

namespace spec {

constexpr int kMkRows = 128;        // MMA M: request rows (rows >= B are zero)
constexpr int kMkTile = 128;        // MMA N: vocabulary rows of W2^T per tile
constexpr int kMkAtomK = 64;        // bf16 along K per 128-byte swizzle atom
constexpr int kMkAtomBytes = 128 * 128;  // one atom of 128 rows x 128 bytes
constexpr int kMkEpiWarps = 8;      // kMkHalves per TMEM lane quarter, taking tiles in turn
constexpr int kMkHalves = kMkEpiWarps / 4;  // epilogue warps per lane quarter
constexpr int kMkParts = 2 * kMkHalves;     // partials per (request, bias CTA)
constexpr int kMkSub = 64;          // sub-block: the columns of a tile one epilogue warp takes
constexpr int kMkRace = kRaceBlock; // race block: four sub-blocks (the blocks of every draw)
constexpr int kMkThreads = 32 * (2 + kMkEpiWarps);  // warp 0 TMA, warp 1 MMA, then the epilogue
constexpr int kMkMaxR = 256;
constexpr int kMkSlots = 4;         // accumulators: tile t in slot t % 4
constexpr int kMkTmemCols = kMkSlots * kMkTile;  // 512 fp32 columns
constexpr int kPickThreads = 1024;  // level 2: 32 warps x 8 entries = one race block

struct alignas(16) MkPartial {
  float m, s;     // softmax statistics of the CTA's columns (s relative to fl(m*c2))
  float L;        // tau = 0: the max
  int32_t idx;    // tau = 0: lowest argmax (INT_MAX: none)
  float M;        // unused
  int32_t flags;  // bit0: NaN or +inf
  int32_t pad[2];
};

struct MarkovLaunch {
  const __nv_bfloat16* U;    // [B, K, V]
  const __nv_bfloat16* W1;   // [V, r]
  const __nv_bfloat16* W2T;  // [V, r]: row v = column v of W2
  int r, B, K, V, step;
  float tau, c2, inv_t;
  const uint64_t* seeds;
  const uint64_t* request_ids;
  const int64_t* pos_base;
  const int32_t* x0;
  __nv_bfloat16* E;  // [128, r]: W1 at the previous drafts
  MkPartial* part;   // [B][G][kMkParts]: per bias CTA, per epilogue group and column half
  float2* sub;       // [B][nsub_pad]: per 64-column sub-block (max, sum relative to fl(max*c2)), tau > 0
  int nsub, nsub_pad;
  int G;
  uint32_t* req_bad;  // [B]
  int32_t* drafts;
  float* conf;
  float* scores;
  float* row_stats;
  int32_t* status;
  bool u_vec;
};

// ---------------------------------------------------------------------------
// PTX wrappers: mbarrier, TMA, tcgen05
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return done != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Wait for the phase with parity `parity`; false (and SPEC_ERR_TIMEOUT) after
// about a second.  The bounded loop is out of line; the first try is not.
__device__ __noinline__ bool mbar_wait_slow(uint64_t* bar, uint32_t parity, int32_t* status) {
  const uint64_t t0 = global_ns();
  for (uint32_t it = 0;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 255u && global_ns() - t0 > 1000000000ull) {
      report(status, SPEC_ERR_TIMEOUT);
      return false;
    }
  }
}
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int32_t* status) {
  return mbar_try_wait(bar, parity) || mbar_wait_slow(bar, parity, status);
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// K-major operand in 128-byte swizzled atoms (rows of 128 bytes, 8-row
// groups 1024 bytes apart): start address, SBO = 1024, descriptor version 1,
// layout SWIZZLE_128B.
__device__ __forceinline__ uint64_t umma_desc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)1 << 16;             // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;   // stride byte offset: next 8-row group
  d |= (uint64_t)1 << 46;             // descriptor version
  d |= (uint64_t)2 << 61;             // SWIZZLE_128B
  return d;
}
// kind::f16 instruction descriptor: fp32 accumulator, bf16 A and B, both
// K-major, N and M.
__host__ __device__ constexpr uint32_t umma_idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t accum) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(idesc), "r"(accum)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32 consecutive fp32 columns of this warp's 32 TMEM lanes (one per thread).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int k = 0; k < 32; ++k) v[k] = __uint_as_float(r[k]);
}

// ---------------------------------------------------------------------------
// Level-1 keys as in draft.cu (log2 domain, compared as differences)
// ---------------------------------------------------------------------------
struct MkKey {
  float L, M;
  int32_t idx;
};
__device__ __forceinline__ bool mk_better(const MkKey& a, const MkKey& b, float c2) {
  if (a.idx == INT_MAX) return false;
  if (b.idx == INT_MAX) return true;
  const float lhs = a.L - b.L, rhs = c2 * (a.M - b.M);
  return lhs < rhs || (lhs == rhs && a.idx < b.idx);
}
__device__ __forceinline__ SoftState mk_merge(SoftState a, SoftState b, float c2) {
  if (b.m > a.m) {
    const SoftState t = a;
    a = b;
    b = t;
  }
  if (b.m == -INFINITY) return a;
  a.s = a.s + b.s * ex2_approx(b.m * c2 - a.m * c2);
  return a;
}
__device__ __forceinline__ float mk_lg2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ---------------------------------------------------------------------------
// The bias and level-1 pass of one position
// ---------------------------------------------------------------------------
template <bool kGreedy>
__global__ void __launch_bounds__(kMkThreads, 1)
    markov_bias_kernel(const __grid_constant__ CUtensorMap tmE, const __grid_constant__ CUtensorMap tmW,
                       const MarkovLaunch p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int nk = p.r / kMkAtomK;
  uint8_t* sA = smem;                          // nk atoms
  uint8_t* sB = smem + nk * kMkAtomBytes;      // 2 stages of nk atoms
  // Tile t uses smem stage t & 1 and accumulator slot t & 3, so that every
  // waiter of a barrier sees its phases one after another (a parity wait two
  // phases behind would alias).
  __shared__ uint64_t bar_a, bar_full[2], bar_mma[kMkSlots], bar_free[kMkSlots];
  __shared__ uint32_t tmem_base_sh;
  __shared__ int abort_flag;
  volatile int& abort_sh = abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ntiles = (p.V + kMkTile - 1) / kMkTile;
  const int T = ntiles > (int)blockIdx.x ? (ntiles - 1 - (int)blockIdx.x) / p.G + 1 : 0;  // tile t: blockIdx.x + t G
  // Epilogue warps: TMEM lane quarter q = warp % 4, group eh = the tiles with
  // t % kMkHalves == eh.  With B <= 64 the operand's rows 64..127 repeat rows 0..63,
  // so every request row sits in two quarters: quarters 0-1 take a tile's
  // columns 0..63 and quarters 2-3 its columns 64..127, and all four SM
  // sub-partitions share the epilogue.  With B > 64 a warp takes its 32 rows
  // over all 128 columns.
  const bool dup = p.B <= 64;
  const bool epi = warp >= 2;
  const int q = warp & 3;
  const int eh = (warp - 2) >> 2;
  const int row_q = dup ? (q & 1) : q;       // the quarter of request rows this warp serves
  const int col_half = dup ? (q >> 1) : 0;   // with dup: columns [64 col_half, 64 col_half + 64)
  const bool epi_active = epi && 32 * row_q < p.B;
  const int n_epi = dup ? (p.B > 32 ? 4 : 2) : (p.B + 31) / 32;  // readers of each tile

  // The next kernel (this position's pick) may launch now; its CTAs do not
  // fit beside a bias CTA (registers), so they start as bias CTAs exit.
  pdl_launch_dependents();
  if (threadIdx.x == 0) {
    mbar_init(&bar_a, 1);
    for (int s = 0; s < 2; ++s) mbar_init(&bar_full[s], 1);
    for (int k = 0; k < kMkSlots; ++k) {
      mbar_init(&bar_mma[k], 1);
      mbar_init(&bar_free[k], (uint32_t)n_epi);
    }
    abort_sh = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base_sh)),
                 "r"(kMkTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_sh;

  if (warp == 0) {
    // ---- TMA producer ----
    if (lane == 0 && T > 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmE)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmW)) : "memory");
      // W2^T and U are inputs of the whole draw, complete before its first
      // kernel started: the first two tiles load while the previous
      // position's pick runs.  E is that pick's output.
      const int t_pre = T < 2 ? T : 2;
      for (int t = 0; t < t_pre; ++t) {
        const int v0 = ((int)blockIdx.x + t * p.G) * kMkTile;
        mbar_expect_tx(&bar_full[t], (uint32_t)(nk * kMkAtomBytes));
        for (int a = 0; a < nk; ++a)
          tma_load_2d(sB + (t * nk + a) * kMkAtomBytes, &tmW, a * kMkAtomK, v0, &bar_full[t]);
      }
      pdl_wait_prerequisites();
      mbar_expect_tx(&bar_a, (uint32_t)(nk * kMkAtomBytes));
      for (int a = 0; a < nk; ++a) tma_load_2d(sA + a * kMkAtomBytes, &tmE, a * kMkAtomK, 0, &bar_a);
      for (int t = t_pre; t < T; ++t) {
        const int s = t & 1;
        // the stage's previous tile (t - 2) has been consumed by its MMA
        if (!mbar_wait(&bar_mma[(t - 2) & 3], (uint32_t)(((t - 2) >> 2) & 1), p.status)) {
          abort_sh = 1;
          break;
        }
        if (abort_sh) break;
        const int v0 = ((int)blockIdx.x + t * p.G) * kMkTile;
        mbar_expect_tx(&bar_full[s], (uint32_t)(nk * kMkAtomBytes));
        for (int a = 0; a < nk; ++a)
          tma_load_2d(sB + (s * nk + a) * kMkAtomBytes, &tmW, a * kMkAtomK, v0, &bar_full[s]);
      }
    }
  } else if (warp == 1) {
    // ---- MMA issuer ----
    int issued = 0;
    if (lane == 0 && T > 0) {
      constexpr uint32_t idesc = umma_idesc_bf16(kMkRows, kMkTile);
      if (!mbar_wait(&bar_a, 0u, p.status)) abort_sh = 1;
      for (int t = 0; t < T && !abort_sh; ++t) {
        const int s = t & 1, u = t >> 1, slot = t & 3;
        // the slot's previous tile (t - 4) has been read by the epilogue
        if (t >= kMkSlots && !mbar_wait(&bar_free[slot], (uint32_t)(((t >> 2) - 1) & 1), p.status)) {
          abort_sh = 1;
          break;
        }
        if (!mbar_wait(&bar_full[s], (uint32_t)(u & 1), p.status)) {
          abort_sh = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(slot * kMkTile);
        for (int kk = 0; kk < p.r / 16; ++kk) {
          const uint32_t koff = (uint32_t)((kk >> 2) * kMkAtomBytes + (kk & 3) * 32);
          const uint64_t da = umma_desc_sw128(smem_u32(sA) + koff);
          const uint64_t db = umma_desc_sw128(smem_u32(sB + s * nk * kMkAtomBytes) + koff);
          umma_bf16(d, da, db, idesc, kk > 0 ? 1u : 0u);
        }
        umma_commit(&bar_mma[slot]);
        issued = t + 1;
      }
      // what was issued completes before the TMEM is freed
      if (issued > 0) mbar_wait(&bar_mma[(issued - 1) & 3], (uint32_t)(((issued - 1) >> 2) & 1), p.status);
    }
    __syncwarp();
  } else if (epi_active) {
    // ---- epilogue: one request row per thread ----
    const int row = 32 * row_q + lane;
    const bool valid = row < p.B;
    const size_t urow = ((size_t)(valid ? row : 0) * p.K + p.step) * (size_t)p.V;
    const int nblk = dup ? 1 : 2;            // sub-blocks of a tile this warp takes
    const int blk0 = dup ? col_half : 0;
    SoftState st{-INFINITY, 0.0f};
    ArgState g{-INFINITY, INT_MAX};
    int32_t flags = 0;
    bool aborted = false;
    // A lane reads 128 consecutive bytes of its own row of U in 16-byte
    // loads (one 64-column sub-block); the loads allocate in L1, so each
    // 32-byte sector crosses from L2 once.
    uint4 uw[8];
    auto load_u = [&](int vb) {
#pragma unroll
      for (int h = 0; h < 8; ++h) {
        const int v = vb + 8 * h;
        if (valid && p.u_vec && v + 8 <= p.V) {
          uw[h] = __ldg(reinterpret_cast<const uint4*>(p.U + urow + v));
        } else {
          uint32_t e[8];
#pragma unroll
          for (int j = 0; j < 8; ++j)
            e[j] = (valid && v + j < p.V) ? (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(p.U) + urow + v + j)
                                          : 0xFF80u;  // -inf past V
          uw[h] = make_uint4(e[0] | e[1] << 16, e[2] | e[3] << 16, e[4] | e[5] << 16, e[6] | e[7] << 16);
        }
      }
    };
    for (int t = eh; t < T; t += kMkHalves) {
      const int slot = t & 3;
      const int v0 = ((int)blockIdx.x + t * p.G) * kMkTile;
      // the warp's first sub-block of U, fetched before the accumulator wait
      load_u(v0 + kMkSub * blk0);
      // the warp's next tile of U, into L2 while this one is processed
      if (valid && t + kMkHalves < T) {
        const int vn = ((int)blockIdx.x + (t + kMkHalves) * p.G) * kMkTile + kMkSub * blk0;
        const int ve = min(vn + kMkSub * nblk, p.V) - 1;
        if (vn < p.V)
          for (int x = vn; x <= ve; x += 64) {
            asm volatile("prefetch.global.L2 [%0];" ::"l"(p.U + urow + x));
            asm volatile("prefetch.global.L2 [%0];" ::"l"(p.U + urow + min(x + 63, ve)));
          }
      }
      const bool ok = __all_sync(0xFFFFFFFFu, mbar_wait(&bar_mma[slot], (uint32_t)((t >> 2) & 1), p.status));
      if (!ok) {
        aborted = true;
        break;
      }
      tc_fence_after();
      for (int cb = 0; cb < nblk; ++cb) {
        const int bcol = kMkSub * (blk0 + cb);  // the sub-block's first column in the tile
        const int sb = (v0 + bcol) / kMkSub;
        if (cb > 0) load_u(v0 + bcol);  // B > 64: the warp's second sub-block
        SoftState blk{-INFINITY, 0.0f};
#pragma unroll
        for (int ch = 0; ch < kMkSub / 32; ++ch) {
          float l[32];
          tmem_ld32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(slot * kMkTile + bcol + 32 * ch), l);
          float cmax = -INFINITY;
#pragma unroll
          for (int k = 0; k < 32; ++k) {
            const uint4& w4 = uw[(32 * ch + k) >> 3];
            const int e = k & 7;
            const uint32_t word = e < 2 ? w4.x : e < 4 ? w4.y : e < 6 ? w4.z : w4.w;
            l[k] += (e & 1) ? bf16_hi(word) : bf16_lo(word);  // -inf past V (U reads -inf there, the bias is 0)
            cmax = fmaxf(cmax, l[k]);
          }
          if (!valid) continue;
          if (cmax == INFINITY) flags |= 1;
          if (kGreedy && cmax > -INFINITY && (g.idx == INT_MAX || cmax > g.v || (cmax == g.v && v0 + bcol + 32 * ch < g.idx))) {
            int first = INT_MAX;
#pragma unroll
            for (int k = 31; k >= 0; --k)
              if (l[k] == cmax) first = v0 + bcol + 32 * ch + k;
            if (g.idx == INT_MAX || cmax > g.v || first < g.idx) g = ArgState{cmax, first};
          }
          if (cmax > -INFINITY && cmax < INFINITY) {
            const float M2 = cmax * p.c2;
            float cs = 0.0f;
#pragma unroll
            for (int k = 0; k < 32; ++k) cs += ex2_approx(__fmaf_rn(l[k], p.c2, -M2));
            if (cs != cs) flags |= 1;  // a NaN entry
            else blk = mk_merge(blk, SoftState{cmax, cs}, p.c2);
          } else if (cmax != cmax) {
            flags |= 1;
          }
        }
        if (!valid) continue;
        // the sub-block is complete: its statistics for the pick's level 1
        st = mk_merge(st, blk, p.c2);
        if (!kGreedy && sb < p.nsub) p.sub[(size_t)row * p.nsub_pad + sb] = make_float2(blk.m, blk.s);
      }
      // the accumulator is read: the MMA may overwrite it
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar_free[slot]);
    }
    pdl_wait_prerequisites();  // the previous position's pick has read the partials
    if (valid && !aborted) {
      MkPartial o{};
      o.m = st.m;
      o.s = st.s;
      o.L = kGreedy ? g.v : 0.0f;
      o.idx = kGreedy ? g.idx : INT_MAX;
      o.flags = flags;
      MkPartial* dstp = p.part + ((size_t)row * p.G + blockIdx.x) * kMkParts + 2 * eh;
      dstp[col_half] = o;
      if (!dup) {  // this warp covered both column halves
        MkPartial none{};
        none.m = -INFINITY;
        none.L = kGreedy ? -INFINITY : INFINITY;
        none.idx = INT_MAX;
        dstp[1] = none;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kMkTmemCols) : "memory");
  }
}

// ---------------------------------------------------------------------------
// The draw of one position: merge, level 1, level 2, outputs, next E
// ---------------------------------------------------------------------------
// MkKey of the best of two candidates, over a warp (xor butterfly).
__device__ __forceinline__ MkKey mk_warp_best(MkKey k, float c2) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const MkKey ok{__shfl_xor_sync(0xFFFFFFFFu, k.L, o), __shfl_xor_sync(0xFFFFFFFFu, k.M, o),
                   __shfl_xor_sync(0xFFFFFFFFu, k.idx, o)};
    if (mk_better(ok, k, c2)) k = ok;
  }
  return k;
}

template <bool kGreedy>
__global__ void __launch_bounds__(kPickThreads, 1) markov_pick_kernel(const MarkovLaunch p) {
  constexpr int kW = kPickThreads / 32;
  __shared__ __align__(16) __nv_bfloat16 sh_e[kMkMaxR];
  __shared__ float sh_l[kMkRace];
  __shared__ KeyState sh_red[kW];
  __shared__ MkPartial sh_part[kW];
  __shared__ MkKey sh_key[kW];
  __shared__ float sh_m, sh_S;
  __shared__ int sh_idx, sh_bad;
  const int i = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // inputs of the whole draw, read before the wait
  const long long pos = __ldg(reinterpret_cast<const long long*>(p.pos_base) + i);
  const uint64_t req = __ldg(reinterpret_cast<const unsigned long long*>(p.request_ids) + i);
  const uint64_t seed = __ldg(reinterpret_cast<const unsigned long long*>(p.seeds) + i);
  const uint32_t position = (uint32_t)(pos + p.step + 1);
  // the next position's bias kernel may launch now: it prefetches its first
  // W2^T tiles and waits for this grid before it reads E
  pdl_launch_dependents();
  pdl_wait_prerequisites();
  // this position's operand row, kept in a register until level 2 (a store
  // to shared memory now would hold the thread's next loads back a round trip)
  const __nv_bfloat16 e_own = (int)threadIdx.x < p.r ? p.E[(size_t)i * p.r + threadIdx.x] : __float2bfloat16(0.0f);

  // a bad request stays bad: the flag of the positions before, read now
  const uint32_t was_bad = threadIdx.x == 0 ? __ldcg(p.req_bad + i) : 0u;

  // ---- tau > 0: this thread's first race block (four 64-column
  // sub-blocks, two 16-byte loads), loaded together with the partials below ----
  const int nb = (p.V + kMkRace - 1) / kMkRace;  // race blocks
  const float4* subrow = reinterpret_cast<const float4*>(p.sub + (size_t)i * p.nsub_pad);
  const float4 kNoSub = make_float4(-INFINITY, 0.f, -INFINITY, 0.f);
  float4 sq0 = kNoSub, sq1 = kNoSub;
  if (!kGreedy) {
    const int b = threadIdx.x;
    if (b < nb) sq0 = __ldcg(subrow + 2 * b);
    if (b < nb && 4 * b + 2 < p.nsub) sq1 = __ldcg(subrow + 2 * b + 1);
  }

  // ---- merge the kMkParts * G partials of the bias CTAs ----
  {
    SoftState st{-INFINITY, 0.0f};
    ArgState g{-INFINITY, INT_MAX};
    int32_t f = 0;
    const int n = kMkParts * p.G;
    const uint4* src = reinterpret_cast<const uint4*>(p.part + (size_t)i * n);
    for (int c = threadIdx.x; c < n; c += kPickThreads) {
      const uint4 lo = __ldcg(src + 2 * c), hi = __ldcg(src + 2 * c + 1);
      st = soft_merge(st, SoftState{__uint_as_float(lo.x), __uint_as_float(lo.y)}, p.c2);
      f |= (int32_t)hi.y;
      if (kGreedy) {
        const ArgState a{__uint_as_float(lo.z), (int)lo.w};
        if (arg_better(a, g)) g = a;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      st = soft_merge(st, SoftState{__shfl_xor_sync(0xFFFFFFFFu, st.m, o), __shfl_xor_sync(0xFFFFFFFFu, st.s, o)},
                      p.c2);
      if (kGreedy) {
        const ArgState og{__shfl_xor_sync(0xFFFFFFFFu, g.v, o), __shfl_xor_sync(0xFFFFFFFFu, g.idx, o)};
        if (arg_better(og, g)) g = og;
      }
    }
    f = (int32_t)__reduce_or_sync(0xFFFFFFFFu, (unsigned)f);
    if (lane == 0) {
      MkPartial w{};
      w.m = st.m;
      w.s = st.s;
      w.L = g.v;
      w.idx = g.idx;
      w.flags = f;
      sh_part[warp] = w;
    }
  }

  // ---- level 1 (tau > 0): the key of every 256-entry block from its four
  // 64-column sub-blocks, log2 E_b - log2 sum_b against the block's max; a
  // block per thread ----
  if (!kGreedy) {
    MkKey best{INFINITY, 0.0f, INT_MAX};
    for (int b = threadIdx.x; b < nb; b += kPickThreads) {
      if (b != (int)threadIdx.x) {  // blocks past the first: loaded here
        sq0 = __ldcg(subrow + 2 * b);
        sq1 = 4 * b + 2 < p.nsub ? __ldcg(subrow + 2 * b + 1) : kNoSub;
      }
      const uint4 rq = philox(draw_counter(position, req, SPEC_PURPOSE_DRAFT, (uint32_t)(b >> 2)), (uint32_t)seed,
                              (uint32_t)(seed >> 32));
      const int e = b & 3;
      const uint32_t word = e == 0 ? rq.x : e == 1 ? rq.y : e == 2 ? rq.z : rq.w;
      // sub-blocks 4b .. 4b+3 in order; those at or past nsub add nothing
      SoftState blk{-INFINITY, 0.0f};
      blk = mk_merge(blk, SoftState{sq0.x, sq0.y}, p.c2);
      if (4 * b + 1 < p.nsub) blk = mk_merge(blk, SoftState{sq0.z, sq0.w}, p.c2);
      if (4 * b + 2 < p.nsub) blk = mk_merge(blk, SoftState{sq1.x, sq1.y}, p.c2);
      if (4 * b + 3 < p.nsub) blk = mk_merge(blk, SoftState{sq1.z, sq1.w}, p.c2);
      if (blk.m > -INFINITY && blk.s > 0.0f && isfinite(blk.s)) {
        const float E = -log1pf(-((float)race_m(word) * 0x1p-24f));
        const MkKey cand{mk_lg2(E) - mk_lg2(blk.s), blk.m, b};
        if (mk_better(cand, best, p.c2)) best = cand;
      }
    }
    best = mk_warp_best(best, p.c2);
    if (lane == 0) sh_key[warp] = best;
  }
  if ((int)threadIdx.x < p.r) sh_e[threadIdx.x] = e_own;
  __syncthreads();
  if (threadIdx.x < 32) {
    // warp 0 merges the warps' results
    SoftState st{-INFINITY, 0.0f};
    MkKey best{INFINITY, 0.0f, INT_MAX};
    ArgState g{-INFINITY, INT_MAX};
    int32_t f = 0;
    if (lane < kW) {
      const MkPartial& o = sh_part[lane];
      st = SoftState{o.m, o.s};
      f = o.flags;
      g = ArgState{o.L, o.idx};
      if (!kGreedy) best = sh_key[lane];
    }
#pragma unroll
    for (int o = kW / 2; o > 0; o >>= 1) {
      st = soft_merge(st, SoftState{__shfl_xor_sync(0xFFFFFFFFu, st.m, o), __shfl_xor_sync(0xFFFFFFFFu, st.s, o)},
                      p.c2);
      const ArgState og{__shfl_xor_sync(0xFFFFFFFFu, g.v, o), __shfl_xor_sync(0xFFFFFFFFu, g.idx, o)};
      if (arg_better(og, g)) g = og;
    }
    if (!kGreedy) best = mk_warp_best(best, p.c2);
    f = (int32_t)__reduce_or_sync(0xFFFFFFFFu, (unsigned)f);
    if (lane == 0) {
      sh_m = st.m;
      sh_S = st.s;
      sh_idx = kGreedy ? g.idx : best.idx;
      sh_bad = (f || was_bad || !(st.m > -INFINITY) || !(st.s > 0.0f) || !isfinite(st.s) || sh_idx == INT_MAX)
                   ? 1 : 0;
    }
  }
  __syncthreads();
  const bool bad = sh_bad != 0;
  const float M2 = sh_m * p.c2;
  int z = -1;
  float lz = sh_m;
  if (!bad) {
    if (kGreedy) {
      z = sh_idx;
    } else {
      // level 2: the winning block's 256 logits recomputed (U + E . W2^T
      // row).  Warp w takes entries 8w..8w+7 of the block; lane l multiplies
      // the r-slice 8l..8l+7 of each (one coalesced 16-byte load per entry,
      // all issued at once), and a transposed butterfly leaves entry
      // 8w + l / 4's dot product in lanes 4 (l / 4)..4 (l / 4) + 3.
      const int b = sh_idx;
      const int v_base = b * kMkRace + 8 * warp;
      const int v = v_base + (lane >> 2);
      const bool owner = (lane & 3) == 0;
      const float u_v = (owner && v < p.V) ? load_elem(p.U + ((size_t)i * p.K + p.step) * (size_t)p.V + v) : 0.0f;
      float part[8];
      {
        const bool has = 8 * lane < p.r;
        uint4 e8 = make_uint4(0u, 0u, 0u, 0u);
        if (has) e8 = *reinterpret_cast<const uint4*>(sh_e + 8 * lane);
        const uint32_t ee[4] = {e8.x, e8.y, e8.z, e8.w};
        uint4 w8[8];
#pragma unroll
        for (int j = 0; j < 8; ++j)
          w8[j] = (has && v_base + j < p.V)
                      ? __ldg(reinterpret_cast<const uint4*>(p.W2T + (size_t)(v_base + j) * p.r) + lane)
                      : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const uint32_t ww[4] = {w8[j].x, w8[j].y, w8[j].z, w8[j].w};
          float acc = 0.0f;
#pragma unroll
          for (int h = 0; h < 4; ++h) {
            acc = fmaf(bf16_lo(ee[h]), bf16_lo(ww[h]), acc);
            acc = fmaf(bf16_hi(ee[h]), bf16_hi(ww[h]), acc);
          }
          part[j] = acc;
        }
      }
      // transposed butterfly over lane bits 4, 3, 2 (4 + 2 + 1 exchanges),
      // then plain sums over bits 1 and 0
#pragma unroll
      for (int n = 8, o = 16; n > 1; n >>= 1, o >>= 1) {
        const bool hi = (lane & o) != 0;
#pragma unroll
        for (int j = 0; j < n / 2; ++j) {
          const float send = hi ? part[j] : part[j + n / 2];
          const float keep = hi ? part[j + n / 2] : part[j];
          part[j] = keep + __shfl_xor_sync(0xFFFFFFFFu, send, o);
        }
      }
      part[0] += __shfl_xor_sync(0xFFFFFFFFu, part[0], 2);
      part[0] += __shfl_xor_sync(0xFFFFFFFFu, part[0], 1);
      KeyState e{INFINITY, INT_MAX};
      float l = -INFINITY;
      if (owner && v < p.V) {
        l = u_v + part[0];
        const float w = ex2_approx(__fmaf_rn(l, p.c2, -M2));
        const uint4 rw =
            philox(draw_counter(position, req, SPEC_PURPOSE_DRAFT_IN_BLOCK, (uint32_t)(v >> 2)), (uint32_t)seed,
                   (uint32_t)(seed >> 32));
        const uint32_t word = (v & 3) == 0 ? rw.x : (v & 3) == 1 ? rw.y : (v & 3) == 2 ? rw.z : rw.w;
        if (w > 0.0f) e = KeyState{race_key(race_m(word), w), v};
      }
      if (owner) sh_l[8 * warp + (lane >> 2)] = l;
      // the lowest key over the CTA
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const KeyState other{__shfl_xor_sync(0xFFFFFFFFu, e.key, o), __shfl_xor_sync(0xFFFFFFFFu, e.idx, o)};
        if (key_better(other, e)) e = other;
      }
      if (lane == 0) sh_red[warp] = e;
      __syncthreads();
      if (warp == 0) {
        KeyState a = lane < kW ? sh_red[lane] : KeyState{INFINITY, INT_MAX};
#pragma unroll
        for (int o = kW / 2; o > 0; o >>= 1) {
          const KeyState other{__shfl_xor_sync(0xFFFFFFFFu, a.key, o), __shfl_xor_sync(0xFFFFFFFFu, a.idx, o)};
          if (key_better(other, a)) a = other;
        }
        if (lane == 0) sh_idx = a.idx == INT_MAX ? -1 : a.idx;
      }
      __syncthreads();
      z = sh_idx;
      if (z >= 0) lz = sh_l[z - b * kMkRace];
    }
  }
  // the next position's operand row: W1 at this draft
  if (p.step + 1 < p.K && (int)threadIdx.x < p.r) {
    const __nv_bfloat16 w = p.W1[(size_t)(bad || z < 0 ? 0 : z) * p.r + threadIdx.x];
    p.E[(size_t)i * p.r + threadIdx.x] = w;
    if (p.B <= 64) p.E[(size_t)(i + 64) * p.r + threadIdx.x] = w;  // the repeated rows
  }
  if (threadIdx.x != 0) return;
  const size_t o = (size_t)i * p.K + p.step;
  if (bad || z < 0) {
    p.req_bad[i] = 1u;
    p.drafts[o] = -1;
    p.conf[o] = 0.0f;
    if (p.row_stats) reinterpret_cast<float2*>(p.row_stats)[o] = make_float2(0.0f, 0.0f);
  } else {
    p.drafts[o] = z;
    p.conf[o] = exp2f(fmaf(lz, p.c2, -M2)) / sh_S;
    if (p.row_stats) {
      const float resid = fmaf(sh_m, p.c2, -M2);
      reinterpret_cast<float2*>(p.row_stats)[o] = make_float2(sh_m * p.inv_t, (log2f(sh_S) - resid) * 0.69314718055994531f);
    }
  }
  if (p.step + 1 < p.K) return;
  // ---- the last position: a bad request's outputs, the scores ----
  const bool req_bad = p.req_bad[i] != 0u;
  if (req_bad) {
    p.req_bad[i] = 0u;  // leave the workspace zeroed for the next call
    report(p.status, SPEC_ERR_BAD_INPUT);
    for (int k = 0; k < p.K; ++k) {
      p.drafts[(size_t)i * p.K + k] = -1;
      p.conf[(size_t)i * p.K + k] = 0.0f;
      if (p.row_stats) reinterpret_cast<float2*>(p.row_stats)[(size_t)i * p.K + k] = make_float2(0.0f, 0.0f);
    }
  }
  if (p.scores) {
    float* sc = p.scores + (size_t)i * (p.K + 1);
    float run = 1.0f;
    sc[0] = run;
    for (int k = 0; k < p.K; ++k) {
      run = req_bad ? 0.0f : __fmul_rn(run, p.conf[(size_t)i * p.K + k]);
      sc[k + 1] = run;
    }
  }
}

// The first position's operand: W1 at the last committed tokens; rows past B
// zero (the padding rows of the MMA).  One CTA per row of E.
__global__ void __launch_bounds__(128) markov_begin_kernel(const MarkovLaunch p) {
  const int e = blockIdx.x;                 // row of E
  const int i = p.B <= 64 ? (e & 63) : e;   // its request (rows 64..127 repeat 0..63 when B <= 64)
  pdl_wait_prerequisites();
  int x = 0;
  bool bad = true;
  if (i < p.B) {
    x = __ldg(p.x0 + i);
    const long long pos = __ldg(reinterpret_cast<const long long*>(p.pos_base) + i);
    bad = x < 0 || x >= p.V || pos < 0 || pos + p.K > 0xFFFFFFFFLL;
    if (threadIdx.x == 0 && e == i) p.req_bad[i] = bad ? 1u : 0u;
  }
  for (int j = threadIdx.x; j < p.r; j += blockDim.x)
    p.E[(size_t)e * p.r + j] = (i < p.B && !bad) ? p.W1[(size_t)x * p.r + j] : __float2bfloat16(0.0f);
}

// One warp waits on an mbarrier that nothing arrives at: the bounded wait
// gives up and reports SPEC_ERR_TIMEOUT (spec_check_bounded_wait).
__global__ void __launch_bounds__(32) bounded_wait_check_kernel(int32_t* status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();
  if (threadIdx.x == 0) mbar_wait(&bar, 0u, status);
  __syncwarp();
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

// A [rows, r] bf16 matrix in boxes of 64 (K) x 128 (rows), 128-byte swizzle.
static bool make_map(CUtensorMap* map, const void* base, int r, long long rows) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)r, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)r * 2};
  cuuint32_t box[2] = {(cuuint32_t)kMkAtomK, 128u};
  cuuint32_t estr[2] = {1u, 1u};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct MarkovGeometry {
  int G, nsub, nsub_pad;
  size_t e_off, part_off, sub_off, bad_off, bytes;
};

static MarkovGeometry markov_geometry(int B, int V, int r, int sms) {
  MarkovGeometry g{};
  const int ntiles = (V + kMkTile - 1) / kMkTile;
  g.G = std::max(1, std::min(sms, ntiles));
  // sub-blocks of a row, padded to whole quads of race blocks (16 sub-blocks)
  g.nsub = (V + kMkSub - 1) / kMkSub;
  g.nsub_pad = (g.nsub + 15) / 16 * 16;
  g.e_off = 0;
  g.part_off = ((size_t)kMkRows * r * 2 + 255) / 256 * 256;
  g.sub_off = g.part_off + ((size_t)sizeof(MkPartial) * B * kMkParts * g.G + 255) / 256 * 256;
  g.bad_off = g.sub_off + ((size_t)sizeof(float2) * B * g.nsub_pad + 255) / 256 * 256;
  g.bytes = g.bad_off + ((size_t)4 * B + 255) / 256 * 256;
  return g;
}

static int device_sms() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 1;
  return sms;
}

static bool markov_shape_ok(int B, int K, int V, int r) {
  return B >= 1 && B <= kMkRows && K >= 1 && K <= SPEC_MAX_DRAFTS && V >= 1 && V < SPEC_MAX_VOCAB && r >= kMkAtomK &&
         r <= kMkMaxR && r % kMkAtomK == 0;
}

}  // namespace spec

extern "C" size_t spec_markov_workspace(int B, int K, int V, int r) {
  if (!spec::markov_shape_ok(B, K, V, r)) return 0;
  // sized for up to 1024 SMs, so that the size does not depend on the device
  return spec::markov_geometry(B, V, r, 1024).bytes;
}

extern "C" int spec_markov_draft(const void* U, int u_dtype, const void* W1, const void* W2T, int r,
                                 const int32_t* x0, int B, int K, int V, float tau, const uint64_t* seeds,
                                 const uint64_t* request_ids, const int64_t* pos_base, int32_t* drafts_out,
                                 float* conf_out, float* scores_out, float* row_stats_out, int32_t* status,
                                 void* ws, size_t ws_bytes, cudaStream_t stream) {
  spec::NvtxRange range("spec_markov_draft");
  using namespace spec;
  if (!markov_shape_ok(B, K, V, r) || u_dtype != SPEC_BF16 || !(tau >= 0.0f) || isinf(tau))
    return SPEC_ERR_INVALID_ARG;
  if (!U || !W1 || !W2T || !x0 || !seeds || !request_ids || !pos_base || !drafts_out || !conf_out)
    return SPEC_ERR_INVALID_ARG;
  if (((reinterpret_cast<uintptr_t>(W1) | reinterpret_cast<uintptr_t>(W2T)) & 15u) != 0 ||
      (row_stats_out && (reinterpret_cast<uintptr_t>(row_stats_out) & 7u) != 0))
    return SPEC_ERR_INVALID_ARG;
  const int sms = device_sms();
  const MarkovGeometry g = markov_geometry(B, V, r, std::min(sms, 1024));
  if (!ws || ws_bytes < g.bytes || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return SPEC_ERR_WORKSPACE;
  MarkovLaunch p{};
  p.U = static_cast<const __nv_bfloat16*>(U);
  p.W1 = static_cast<const __nv_bfloat16*>(W1);
  p.W2T = static_cast<const __nv_bfloat16*>(W2T);
  p.r = r;
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
  p.x0 = x0;
  char* base = static_cast<char*>(ws);
  p.E = reinterpret_cast<__nv_bfloat16*>(base + g.e_off);
  p.part = reinterpret_cast<MkPartial*>(base + g.part_off);
  p.sub = reinterpret_cast<float2*>(base + g.sub_off);
  p.nsub = g.nsub;
  p.nsub_pad = g.nsub_pad;
  p.G = g.G;
  p.req_bad = reinterpret_cast<uint32_t*>(base + g.bad_off);
  p.drafts = drafts_out;
  p.conf = conf_out;
  p.scores = scores_out;
  p.row_stats = row_stats_out;
  p.status = status;
  p.u_vec = (reinterpret_cast<uintptr_t>(U) & 15u) == 0 && V % 8 == 0;
  CUtensorMap tmE, tmW;
  if (!make_map(&tmE, p.E, r, kMkRows) || !make_map(&tmW, W2T, r, V)) return SPEC_ERR_CUDA;
  const int nk = r / kMkAtomK;
  const size_t smem = 1024 + (size_t)3 * nk * kMkAtomBytes;
  const bool greedy = tau == 0.0f;
  auto bias = greedy ? markov_bias_kernel<true> : markov_bias_kernel<false>;
  auto pick = greedy ? markov_pick_kernel<true> : markov_pick_kernel<false>;
  if (cudaFuncSetAttribute(bias, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return SPEC_ERR_CUDA;
  cudaError_t err = launch_after_previous(markov_begin_kernel, dim3(kMkRows), dim3(128), 0, stream, p);
  for (int k = 0; k < K && err == cudaSuccess; ++k) {
    p.step = k;
    // one CTA per SM (shared memory): a CTA launched early waits in
    // griddepcontrol.wait for the previous position's pick kernel
    err = launch_after_previous(bias, dim3(g.G), dim3(kMkThreads), smem, stream, tmE, tmW, p);
    if (err == cudaSuccess) err = launch_after_previous(pick, dim3(B), dim3(kPickThreads), 0, stream, p);
  }
  if (err != cudaSuccess || cudaGetLastError() != cudaSuccess) return SPEC_ERR_CUDA;
  return SPEC_OK;
}

extern "C" int spec_check_bounded_wait(int32_t* status, cudaStream_t stream) {
  spec::NvtxRange range("spec_check_bounded_wait");
  if (!status) return SPEC_ERR_INVALID_ARG;
  spec::bounded_wait_check_kernel<<<1, 32, 0, stream>>>(status);
  return cudaGetLastError() == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}
