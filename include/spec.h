/*
 * spec.h -- C ABI of the GB300 batched speculative-verification library
 * (libspec.so, built for sm_103a).
 *
 * One decoding round of the method of arxiv 2607.25852 ("AngelSpec"):
 *   spec_allocate  D-cut batch-level verification-depth allocation and dense
 *                  packing (Section 4.2: Eqs. dcut-score, dcut-expected-advance,
 *                  dcut-budget, dcut-batch-utility, dcut-select; "Packing and
 *                  correctness").
 *   spec_verify    target verification of the packed drafts by rejection
 *                  sampling (Section 1; Eq. mtp-acceptance-tv in Section 2;
 *                  the deterministic-draft, target-only protocol of Section
 *                  4.2), with temperature 0 as the longest argmax prefix.
 *   spec_commit    packing of the committed tokens and of the target hidden
 *                  rows that condition the drafter's next round (Sections 1,
 *                  3.1 and 6).
 *   spec_shard_*   spec_verify for a target whose vocabulary is split over
 *                  tensor-parallel ranks (Section 4.4 serves with TP = 8).
 *   spec_draft     the drafter's side: drafts, their confidences and the
 *                  D-cut scores from the drafter's logits (Section 4.2).
 *   spec_markov_draft
 *                  the Markov head's sequential draw over a block (Section
 *                  3.2): a tensor-core contraction per position.
 *   spec_graph_*, spec_select_round
 *                  a round per candidate budget as CUDA graphs, the budget
 *                  chosen on the device (Section 4.3).
 *
 * Conventions shared by every entry point
 *   - Pointers marked "device" are CUDA device (or managed) memory of the
 *     current device; "host" pointers are ordinary host memory read during
 *     the call.  The caller owns every buffer.  The library never allocates
 *     device memory, never synchronises the stream and never reads device
 *     memory on the host, so every call is stream-ordered on `stream`.
 *   - Argument errors that the host can see return a spec_err code
 *     synchronously and launch nothing.  Data errors found on the device
 *     (bad token ids, NaN logits, confidences outside [0,1], inconsistent
 *     offsets) are reported through `status`, a device int32 that the caller
 *     zero-fills beforehand: the first error code wins (atomic
 *     compare-and-swap), the kernels still run to completion, and the
 *     affected request's outputs are set to defined values (accepted length
 *     0, tokens -1).  No kernel traps or asserts.
 *   - A device-side wait never spins without a bound.
 *   - Element types: SPEC_BF16 (IEEE binary32 truncated to its upper 16 bits)
 *     or SPEC_F32.
 *
 * Random numbers (a reading: the paper does not fix a generator).  Every
 * uniform is drawn from Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11)
 * with key = (lo32(seed_i), hi32(seed_i)) and counter =
 *   (lo32(position), lo32(request_id_i), hi32(request_id_i), purpose<<28 | sub)
 *   SPEC_PURPOSE_ACCEPT: sub = 0; u = (word0 >> 8) * 2^-24 in [0, 1)
 *   SPEC_PURPOSE_SAMPLE:          sub = b >> 2; block variate E_b from word[b & 3]
 *                                 (block b = entries [256 b, 256 b + 256))
 *   SPEC_PURPOSE_SAMPLE_IN_BLOCK: sub = v >> 2; entry variate E'_v from word[v & 3]
 *   SPEC_PURPOSE_DRAFT, SPEC_PURPOSE_DRAFT_IN_BLOCK: the same two variates
 *                  for spec_draft's draw of the drafts
 * where a word x gives E = -ln((2 * (x >> 9) + 1) * 2^-24), the midpoint of
 * one of 2^23 cells of (0, 1), so E > 0;
 * so a round replays bit for bit from (seed, request id, position).
 */
#ifndef SPEC_H_
#define SPEC_H_

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SPEC_ABI_VERSION 1

typedef enum {
  SPEC_OK = 0,
  SPEC_ERR_INVALID_ARG = 1, /* host-visible argument error; nothing launched */
  SPEC_ERR_WORKSPACE = 2,   /* workspace missing, too small or misaligned, or not left zeroed */
  SPEC_ERR_CUDA = 3,        /* a CUDA runtime call failed (e.g. launch) */
  SPEC_ERR_BAD_INPUT = 4,   /* device-detected data error (via *status) */
  SPEC_ERR_TIMEOUT = 5,     /* a bounded device wait gave up (via *status) */
  SPEC_ERR_TOO_LARGE = 6    /* shape needs more than the static scratch of
                               spec_verify_static; nothing launched */
} spec_err;

typedef enum { SPEC_BF16 = 0, SPEC_F32 = 1 } spec_dtype;

/* Entries per level-1 block of the two-level exponential race, the same for
 * every draw of the library (verification, spec_draft, spec_markov_draft). */
#define SPEC_RACE_BLOCK 256

#define SPEC_PURPOSE_ACCEPT 1u
#define SPEC_PURPOSE_SAMPLE 2u
#define SPEC_PURPOSE_SAMPLE_IN_BLOCK 3u
#define SPEC_PURPOSE_DRAFT 4u
#define SPEC_PURPOSE_DRAFT_IN_BLOCK 5u

/* Limits checked on the host (SPEC_ERR_INVALID_ARG beyond them). */
#define SPEC_MAX_VOCAB (1 << 30)       /* V < 2^30 keeps v >> 2 within 28 bits */
#define SPEC_MAX_DRAFTS 255            /* K */
#define SPEC_MAX_ALLOC_POSITIONS 8192  /* B(K+1) for spec_allocate */
#define SPEC_MAX_CANDIDATES 64         /* M for spec_allocate */

/* Human-readable name of a spec_err code (static string). */
const char* spec_error_string(int code);

/* SPEC_ABI_VERSION of the loaded library. */
int spec_version(void);

/* ------------------------------------------------------------------------
 * spec_pointer_device_readable -- 1 if the library's kernels may read `ptr`
 * in place: device or managed memory, or host memory that the device reaches
 * at the same address (pinned by cudaHostAlloc / cudaHostRegister under
 * unified addressing).  0 otherwise (including when no device is present).
 * Inputs marked "device or host-mapped" below may be such host memory: the
 * kernels then read it over the CPU-GPU link (NVLink-C2C on Grace-Blackwell)
 * with no staging copy.  No counterpart in the paper: a property of the
 * hardware the library runs on.
 * ---------------------------------------------------------------------- */
int spec_pointer_device_readable(const void* ptr);

/* ------------------------------------------------------------------------
 * spec_budget_from_ratios -- Eq. (dcut-budget), Section 4.2:
 *   T_m = max(B, ceil(num[m] / den[m] * B * (K + 1)))
 * in exact integer arithmetic, for M ratios (the paper's set is
 * {1/4, 1/2, 3/4, 1}).  Host only.
 *   num, den     host int32 [M]; 0 <= num[m] <= den[m], den[m] > 0.
 *   cand_T_out   host int32 [M].
 * Returns SPEC_OK or SPEC_ERR_INVALID_ARG.
 * ---------------------------------------------------------------------- */
int spec_budget_from_ratios(int B, int K, const int32_t* num, const int32_t* den,
                            int M, int32_t* cand_T_out);

/* ------------------------------------------------------------------------
 * spec_allocate -- D-cut allocation and packing (Section 4.2).
 *   1. s_{i,0} = 1, s_{i,k} = s_{i,k-1} * c_{i,k} as fp32 products taken in
 *      order k = 1..K (Eq. dcut-score).
 *   2. All B(K+1) positions are ranked by s descending, ties toward the
 *      shallower k (the paper's rule), then toward the lower request index.
 *   3. For each candidate budget T_m, the top-T_m positions give keep depths
 *      n_i(T_m) (a contiguous prefix per request) and the utility
 *      U_m = sum_i sum_{k<=n_i} s_{i,k} (Eqs. dcut-expected-advance,
 *      dcut-batch-utility), evaluated exactly as the integer sum of
 *      floor(s * 2^40) and reported as that sum * 2^-40.
 *   4. The chosen budget is the first maximiser of U_m / cost_m (Eq.
 *      dcut-select, fp64 division).
 *   5. Packing: row_offsets = exclusive scan of (n_i + 1); packed row
 *      row_offsets[i] + j carries token last_tokens[i] (j = 0) or
 *      draft_tokens[i][j-1] (j >= 1) at position pos_base[i] + j.
 * Arguments
 *   conf            device fp32 [B, K], row-major: c_{i,k} at [i][k-1].
 *   cand_T          host int32 [M], each in [B, B(K+1)].
 *   cand_cost       host fp64 [M], each finite and > 0 (the profiled
 *                   step latency C(B, rho) of the candidate).
 *   last_tokens     device int32 [B]; draft_tokens device int32 [B, K];
 *   pos_base        device int64 [B] (position of row 0 of each request).
 *   depth_out       device int32 [B]; row_offsets_out device int32 [B+1];
 *   packed_tokens_out device int32 [B(K+1)], packed_pos_out device int64
 *                   [B(K+1)]: rows past the chosen budget are set to -1.
 *   chosen_T_out    device int32 [1]; utility_out device fp64 [M] or NULL.
 *   status          device int32 [1] (see conventions).
 *   ws, ws_bytes    unused (spec_allocate_workspace returns 0); may be NULL.
 * Limits: 1 <= B, 0 <= K <= SPEC_MAX_DRAFTS, B(K+1) <= SPEC_MAX_ALLOC_POSITIONS,
 * 1 <= M <= SPEC_MAX_CANDIDATES.  A confidence that is NaN or outside [0, 1]
 * counts as 0 and sets SPEC_ERR_BAD_INPUT.
 * ---------------------------------------------------------------------- */
size_t spec_allocate_workspace(int B, int K, int M);
int spec_allocate(const float* conf, int B, int K, const int32_t* cand_T,
                  const double* cand_cost, int M, const int32_t* last_tokens,
                  const int32_t* draft_tokens, const int64_t* pos_base,
                  int32_t* depth_out, int32_t* row_offsets_out,
                  int32_t* packed_tokens_out, int64_t* packed_pos_out,
                  int32_t* chosen_T_out, double* utility_out, int32_t* status,
                  void* ws, size_t ws_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * spec_verify -- batched verification (Section 1: rejection sampling with
 * the target unchanged; Eq. mtp-acceptance-tv; Section 4.2: deterministic-
 * draft, target-only protocol when q is NULL).
 * For request i with n = n_i kept drafts z_1..z_n and logits rows
 * l_0..l_n (row j verifies draft z_{j+1}; row n is the bonus row):
 *   t == 0: g_j = argmax_v l_j[v] (lowest v on ties);
 *           a = longest prefix with z_{j+1} == g_j; y = g_a.
 *   t  > 0: p_j = softmax(l_j / t); for j = 0..n-1 accept z_{j+1} iff
 *           u_j < min(1, p_j(z_{j+1}) / q_j(z_{j+1}))   (q_j(z) = 0 gives 1
 *           if p_j(z) > 0); at the first rejection a = j and y is drawn from
 *           max(0, p_a - q_a) (from p_a if that is identically zero); if all
 *           n are accepted, a = n and y is drawn from p_n.  The draw is a
 *           two-level exponential race: with blocks of 256 consecutive
 *           entries and W_b = sum_{v in b} w_v, first
 *           b* = argmin_{W_b > 0} E_b / W_b, then
 *           y = argmin_{v in b*, w_v > 0} E'_v / w_v (lowest index on ties
 *           at both levels): an exact sampler of w / sum(w), since
 *           P(b*) = W_b / W and P(y | b*) = w_y / W_b.
 *   out_tokens[i] = z_1..z_a, y, then -1 up to K+1 entries.
 * Arguments
 *   logits          device or host-mapped [R, V] of logits_dtype, rows of
 *                   request i at row_offsets[i] .. row_offsets[i] + n_i.
 *   row_offsets     device int32 [B+1] (from spec_allocate) or NULL, meaning
 *                   row_offsets[i] = i(K+1) and R = B(K+1).
 *   depth           device int32 [B] (n_i in [0, K]) or NULL meaning n_i = K.
 *                   If row_offsets is given, row_offsets[i+1] - row_offsets[i]
 *                   must equal n_i + 1 (else SPEC_ERR_BAD_INPUT for i).
 *   draft_tokens    device int32 [B, K] (z_{j+1} at [i][j]); may be NULL if K=0.
 *   q               device or host-mapped [B, K, V] of q_dtype (row j of
 *                   request i is the drafter's distribution of z_{j+1}, used
 *                   as stored), or
 *                   NULL: one-hot at the draft token.  Ignored when t == 0.
 *   temperature     t >= 0 and finite.
 *   seeds, request_ids  device uint64 [B]; pos_base device int64 [B]
 *                   (position of row 0; pos_base + n_i < 2^32).
 *   accepted_len_out device int32 [B]; out_tokens device int32 [B, K+1].
 *   p_draft_out     device fp32 [B, K] or NULL: p_j(z_{j+1}) for j < n_i
 *                   (at t == 0: 1 if z_{j+1} == g_j else 0); other entries 0.
 *   row_stats_out   device fp32 [B(K+1), 2] or NULL: per packed row,
 *                   (max_v l/t, ln sum_v exp(l/t - max)); (max_v l, 0) at t == 0.
 *   status          device int32 [1].
 *   ws, ws_bytes    device workspace of at least spec_verify_workspace(B, K, V)
 *                   bytes, 256-byte aligned, zero-filled once before its first
 *                   use; the library leaves it zeroed again after each call.
 *                   Calls that may overlap on the device need separate
 *                   workspaces.
 * Limits: 1 <= B, 0 <= K <= SPEC_MAX_DRAFTS, 1 <= V < SPEC_MAX_VOCAB,
 * logits rows and q rows addressed with 64-bit offsets.
 * ---------------------------------------------------------------------- */
size_t spec_verify_workspace(int B, int K, int V);
int spec_verify(const void* logits, int logits_dtype, const int32_t* row_offsets,
                const int32_t* depth, const int32_t* draft_tokens, const void* q,
                int q_dtype, int B, int K, int V, float temperature,
                const uint64_t* seeds, const uint64_t* request_ids,
                const int64_t* pos_base, int32_t* accepted_len_out,
                int32_t* out_tokens, float* p_draft_out, float* row_stats_out,
                int32_t* status, void* ws, size_t ws_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * spec_verify_static -- spec_verify for callers that cannot allocate device
 * memory.  The paper has no counterpart: this is a deployment convenience.
 * Who needs it: code inside an inference engine that owns all device memory
 * through its own pool and forbids allocations outside it (under a tight
 * budget such an allocation may fail, and it escapes the engine's memory
 * accounting), and code on a latency-critical path that may not call
 * cudaMalloc, which can synchronise the device.
 * Same arguments and results as spec_verify, without ws / ws_bytes: the
 * scratch is a fixed device array of SPEC_STATIC_SCRATCH_BYTES owned by the
 * library, reserved on every GPU that loads it and held until process exit.
 *   - Returns SPEC_ERR_TOO_LARGE, launching nothing, when
 *     spec_verify_workspace(B, K, V) exceeds SPEC_STATIC_SCRATCH_BYTES
 *     (4 MiB holds about 260,000 16-byte row-chunk partials; B=64, K=16,
 *     V=201088 needs spec_verify_workspace(64, 16, 201088) = 87,808
 *     bytes).
 *   - The first call on a device looks up the array's device address (once
 *     per device and CUDA context, with that device current); make that
 *     first call before any stream capture.  A new context on the device
 *     (after cudaDeviceReset, say) is looked up again on its first call.
 *   - Every call on a device shares the one array, which keeps the previous
 *     call's contents; each call clears the part that must start at zero,
 *     on `stream`, after every argument check has passed (a call that
 *     returns an error has queued nothing).
 *     Calls that overlap on the GPU (concurrent streams, or several host
 *     threads) race on the array and give wrong results: serialise them.
 *   - Allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 * ---------------------------------------------------------------------- */
#define SPEC_STATIC_SCRATCH_BYTES (4u << 20)
int spec_verify_static(const void* logits, int logits_dtype, const int32_t* row_offsets,
                       const int32_t* depth, const int32_t* draft_tokens, const void* q,
                       int q_dtype, int B, int K, int V, float temperature,
                       const uint64_t* seeds, const uint64_t* request_ids,
                       const int64_t* pos_base, int32_t* accepted_len_out,
                       int32_t* out_tokens, float* p_draft_out, float* row_stats_out,
                       int32_t* status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * spec_commit -- pack the committed round for the drafter's next step
 * (Section 1: the verified prefix plus one target token is committed;
 * Sections 3.1 and 6: the drafter conditions on target hidden states).
 *   commit_offsets[i] = sum_{i' < i} (a_{i'} + 1), commit_offsets[B] = total.
 *   packed_tokens_out[commit_offsets[i] + j] = out_tokens[i][j], j = 0..a_i.
 *   hidden_out[commit_offsets[i] + j] = hidden[row_offsets[i] + j], j = 0..a_i
 *   (the target states of the context positions that are now committed).
 * Arguments
 *   accepted_len, out_tokens  device int32 [B], [B, K+1] (from spec_verify).
 *   row_offsets     device int32 [B+1] or NULL (= i(K+1)).
 *   hidden          device or host-mapped [R, H] of hidden_dtype, or NULL
 *                   (tokens only).
 *   packed_tokens_out device int32 [B(K+1)] (entries past the total are
 *                   not written); commit_offsets_out device int32 [B+1];
 *   hidden_out      device [B(K+1), H] (worst case) or NULL.
 *   status          device int32 [1]; an accepted length outside [0, K] sets
 *                   SPEC_ERR_BAD_INPUT and is treated as 0.
 * ---------------------------------------------------------------------- */
int spec_commit(const int32_t* accepted_len, const int32_t* out_tokens,
                const int32_t* row_offsets, const void* hidden, int hidden_dtype,
                int B, int K, int H, int32_t* packed_tokens_out,
                int32_t* commit_offsets_out, void* hidden_out, int32_t* status,
                cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Vocabulary-sharded verification -- spec_verify for a target whose output
 * layer is split over S tensor-parallel ranks (the paper serves its target
 * with TP = 8, Section 4.4), each holding the logits (and q) of a contiguous
 * column range [v_begin, v_begin + V_shard) of the vocabulary.  The ranges
 * must cover [0, V) exactly once, in rank order; boundaries are arbitrary
 * (201088 / 8 = 25136 columns per rank, say).  One round:
 *   1. every rank: spec_shard_stats -> its stats records [R] (R = B(K+1));
 *   2. all-gather the S ranks' records in shard order -> [S, R] records;
 *   3. every rank: spec_shard_decide (identical results on every rank);
 *   4. t > 0, every rank: spec_shard_sample -> its race records [B];
 *   5. t > 0: all-gather them in shard order -> [S, B] records;
 *   6. t > 0, every rank: spec_shard_finish writes the sampled tokens.
 * The caller makes the two exchanges (all-gathers of S * R * 32 and
 * S * B * 96 bytes; with every shard on one GPU, the records are simply
 * written side by side).  The random variates are spec_verify's: they depend
 * on vocabulary indices only, and a race block that straddles a shard
 * boundary is completed in spec_shard_finish from the two shards' parts.
 * Results: at t == 0 identical to spec_verify's bit for bit; at t > 0 the
 * shard sums merge in another order than spec_verify's chunks, so
 * probabilities agree within a few fp32 ulps and an acceptance or draw can
 * differ only where its uniform or race keys tie to that precision.
 * Records are opaque, 16-byte aligned device buffers of the sizes below.
 * ---------------------------------------------------------------------- */
#define SPEC_SHARD_STAT_BYTES 32     /* per (shard, packed row) */
#define SPEC_SHARD_DECISION_BYTES 32 /* per request */
#define SPEC_SHARD_RACE_BYTES 96     /* per (shard, request) */

/* Workspace of spec_shard_stats and spec_shard_sample on one rank: 256-byte
 * aligned, zero-filled once before its first use, left zeroed by every call;
 * calls that may overlap on the device need separate workspaces.  0 for an
 * invalid shape. */
size_t spec_shard_workspace(int B, int K, int V_shard);

/* spec_shard_stats -- per packed row, over the shard's columns: (max, sum of
 * exp2(l * c2 - fl(max * c2))) at t > 0 with c2 = log2(e) / t, (max, lowest
 * argmax as a vocabulary index) at t == 0; and, when the row's draft token
 * falls in the shard, its logit and q value there.
 *   logits_shard    device [R, V_shard] of logits_dtype (the shard's columns
 *                   of the rows spec_verify takes), any alignment.
 *   q_shard         device [B, K, V_shard] of q_dtype, or NULL (one-hot q).
 *   row_offsets, depth, draft_tokens, pos_base, temperature, status: as
 *                   spec_verify.
 *   V               the whole vocabulary; v_begin, V_shard this shard's range.
 *   stats_out       device [R] records of SPEC_SHARD_STAT_BYTES.
 * Rows of requests whose depth or offsets are inconsistent are not written
 * (spec_shard_decide reports them).  Returns SPEC_OK, SPEC_ERR_INVALID_ARG,
 * SPEC_ERR_WORKSPACE or SPEC_ERR_CUDA. */
int spec_shard_stats(const void* logits_shard, int logits_dtype, const int32_t* row_offsets,
                     const int32_t* depth, const int32_t* draft_tokens, const void* q_shard,
                     int q_dtype, int B, int K, int V, int v_begin, int V_shard,
                     float temperature, const int64_t* pos_base, void* stats_out,
                     int32_t* status, void* ws, size_t ws_bytes, cudaStream_t stream);

/* spec_shard_decide -- merges the S shards' records of each row (in shard
 * order) and runs spec_verify's decision chain: accepted_len_out, out_tokens
 * (all but the sampled token at t > 0), p_draft_out and row_stats_out as
 * spec_verify writes them.
 *   stats           device [S, R] records gathered from spec_shard_stats.
 *   q_dense         nonzero if the ranks passed q_shard (t > 0).
 *   decisions_out   device [B] records of SPEC_SHARD_DECISION_BYTES; required
 *                   at t > 0, unused at t == 0 (may be NULL).
 * A draft token owned by no shard, or by several, sets SPEC_ERR_BAD_INPUT for
 * its request. */
int spec_shard_decide(const void* stats, int S, const int32_t* row_offsets,
                      const int32_t* depth, const int32_t* draft_tokens, int q_dense, int B,
                      int K, int V, float temperature, const uint64_t* seeds,
                      const uint64_t* request_ids, const int64_t* pos_base,
                      int32_t* accepted_len_out, int32_t* out_tokens, float* p_draft_out,
                      float* row_stats_out, void* decisions_out, int32_t* status,
                      cudaStream_t stream);

/* spec_shard_sample -- t > 0: level 1 of the draw over the race blocks the
 * shard owns whole (with the race over p beside it at a rejection, for the
 * case that no shard has a positive draw weight) and level 2 inside the best
 * of them; for a block cut by a shard boundary, the shard's part of its
 * weight sum and its part's best entry.  Does nothing at t == 0.
 *   decisions       device [B] records from spec_shard_decide.
 *   race_out        device [B] records of SPEC_SHARD_RACE_BYTES. */
int spec_shard_sample(const void* logits_shard, int logits_dtype, const void* q_shard,
                      int q_dtype, const void* decisions, int B, int K, int V, int v_begin,
                      int V_shard, float temperature, const uint64_t* seeds,
                      const uint64_t* request_ids, void* race_out, int32_t* status, void* ws,
                      size_t ws_bytes, cudaStream_t stream);

/* spec_shard_finish -- t > 0: completes the cut blocks (weight sums added in
 * shard order, block variates drawn) and takes the lowest block key over all
 * shards: each request's sampled token in out_tokens.  Does nothing at
 * t == 0.
 *   races           device [S, B] records gathered from spec_shard_sample. */
int spec_shard_finish(const void* races, int S, const void* decisions, int B, int K, int V,
                      float temperature, const uint64_t* seeds, const uint64_t* request_ids,
                      int32_t* accepted_len_out, int32_t* out_tokens, int32_t* status,
                      cudaStream_t stream);

/* ------------------------------------------------------------------------
 * spec_draft -- the drafter's producer step: drafts, token-level confidences
 * and D-cut scores from the drafter's logits in one streaming pass (Section
 * 4.2: D-cut reads the drafter's confidences c_{i,t} and ranks positions by
 * s_{i,k} = prod_{t<=k} c_{i,t}, Eq. dcut-score).  For request i and row k
 * (the drafter's logits for draft z_{k+1}):
 *   q_k = softmax(l_k / tau') with tau' = tau, or 1 when tau == 0;
 *   tau  > 0: z_{k+1} is drawn from q_k by the two-level exponential race of
 *             spec_verify at position pos_base[i] + k + 1, with the variates
 *             of SPEC_PURPOSE_DRAFT (blocks) and SPEC_PURPOSE_DRAFT_IN_BLOCK
 *             (entries);
 *   tau == 0: z_{k+1} = argmax_v l_k[v] (lowest v on ties);
 *   c_{k+1} = q_k(z_{k+1})  (a reading: the paper does not define c);
 *   s_0 = 1, s_k = fl32(s_{k-1} * c_k), the scores spec_allocate forms from
 *   conf.
 * Arguments
 *   logits          device [B, K, V] of logits_dtype, rows contiguous.
 *   seeds, request_ids  device uint64 [B]; pos_base device int64 [B] (the
 *                   position of the last committed token; pos_base + K < 2^32).
 *   drafts_out      device int32 [B, K]; conf_out device fp32 [B, K] (the
 *                   input spec_allocate takes as conf).
 *   scores_out      device fp32 [B, K+1] or NULL.
 *   row_stats_out   device fp32 [B*K, 2] or NULL: per row (max_v l/tau',
 *                   ln sum_v exp(l/tau' - max)).
 *   status          device int32 [1]: a row with a NaN, a +inf or no finite
 *                   logit, or a position past 2^32 - 1, sets
 *                   SPEC_ERR_BAD_INPUT; its request gets drafts -1,
 *                   confidences 0 and scores (1, 0, ..., 0).
 *   ws, ws_bytes    device workspace of at least spec_draft_workspace(B, K, V)
 *                   bytes, 256-byte aligned, zero-filled once before its first
 *                   use; left zeroed after each call.
 * Limits: 1 <= B, 1 <= K <= SPEC_MAX_DRAFTS, 1 <= V < SPEC_MAX_VOCAB.
 * ---------------------------------------------------------------------- */
size_t spec_draft_workspace(int B, int K, int V);
int spec_draft(const void* logits, int logits_dtype, int B, int K, int V, float tau,
               const uint64_t* seeds, const uint64_t* request_ids, const int64_t* pos_base,
               int32_t* drafts_out, float* conf_out, float* scores_out, float* row_stats_out,
               int32_t* status, void* ws, size_t ws_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * spec_markov_draft -- the Markov head's sequential draw (Section 3.2,
 * Eq. dspark-markov; the block factorisation Eq. ar-factorization): for
 * k = 0..K-1, with x_0 the last committed token,
 *   b_k = W1[x_k] W2,  q_k = softmax((U_k + b_k) / tau')  (tau' = tau, or 1),
 *   x_{k+1} ~ q_k by spec_draft's two-level race (blocks of
 *   SPEC_RACE_BLOCK entries, purposes SPEC_PURPOSE_DRAFT / _IN_BLOCK) at
 *   position pos_base + k + 1, argmax at tau == 0: with W1 = 0 the draws
 *   are spec_draft's on the same U;
 *   c_{k+1} = q_k(x_{k+1}); scores as spec_draft.
 * The bias of all B requests is one [B, r] x [r, V] contraction per position,
 * run on the tensor cores (tcgen05, fp32 accumulation): q, c and the row
 * statistics carry its rounding (relative errors of order r * 2^-24 on the
 * bias).
 *   U               device bf16 [B, K, V]: the backbone's base logits.
 *   W1              device bf16 [V, r]; W2T device bf16 [V, r], W2 stored
 *                   transposed (row v = column v of W2), 16-byte aligned.
 *   r               the factorisation's rank: a multiple of 64, 64..256.
 *   x0              device int32 [B]: each request's last committed token.
 *   B <= 128; other arguments and the bad-input rule as spec_draft (an x0
 *   outside [0, V) also makes the request bad).
 *   ws, ws_bytes    spec_markov_workspace(B, K, V, r) bytes, 256-aligned, no
 *                   zeroing needed.
 * ---------------------------------------------------------------------- */
size_t spec_markov_workspace(int B, int K, int V, int r);
int spec_markov_draft(const void* U, int u_dtype, const void* W1, const void* W2T, int r,
                      const int32_t* x0, int B, int K, int V, float tau, const uint64_t* seeds,
                      const uint64_t* request_ids, const int64_t* pos_base, int32_t* drafts_out,
                      float* conf_out, float* scores_out, float* row_stats_out, int32_t* status,
                      void* ws, size_t ws_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * A whole round per candidate budget as CUDA graphs, the budget chosen on the
 * device (Section 4.3: the reachable verification shapes form a small finite
 * set, so a graph can be captured per (B, rho), and budget selection should
 * leave the critical path instead of synchronising drafting and
 * verification).  Recipe:
 *   1. per candidate T_m: spec_graph_begin_capture(s); enqueue on s what
 *      follows the allocation at that shape (the target forward over T_m
 *      packed rows -- spec_pack_rows stands in for it -- then spec_verify and
 *      spec_commit); spec_graph_end_capture(s, 1, &g[m]);
 *   2. spec_graph_begin_capture(s); spec_allocate(...);
 *      spec_select_round(chosen_T, M, cand_T, g, ...);
 *      spec_graph_end_capture(s, 0, &parent);
 *   3. every round: spec_graph_launch(parent, s).  The selector kernel reads
 *      T* on the device and tail-launches g[m] with cand_T[m] == T*: the
 *      round needs no host round trip between the budget choice and the
 *      verification.  Work enqueued on s after the parent waits for the
 *      tail-launched graph too.
 * Graph handles are opaque (cudaGraphExec_t); instantiating a graph allocates
 * what the CUDA driver needs for it (the one exception to "the library never
 * allocates device memory"), released by spec_graph_destroy.
 * ---------------------------------------------------------------------- */
/* Begin capturing `stream` (relaxed capture mode; not the legacy stream). */
int spec_graph_begin_capture(cudaStream_t stream);
/* End the capture and instantiate it; device_launch != 0 instantiates for
 * launch from the device (and uploads it).  *exec_out: the graph handle. */
int spec_graph_end_capture(cudaStream_t stream, int device_launch, void** exec_out);
int spec_graph_launch(void* exec, cudaStream_t stream);
int spec_graph_destroy(void* exec);

/* spec_select_round -- one thread on `stream`: reads *chosen_T (device, as
 * spec_allocate writes it), finds m with cand_T[m] == T*, tail-launches
 * graphs[m] (instantiated with device_launch) and writes m to *launched_out
 * (device int32, or NULL).  Must be captured into a host-launched graph (the
 * device runtime launches graphs only from kernels that run in a graph).  A
 * T* that is not in cand_T sets SPEC_ERR_BAD_INPUT and launches nothing.
 *   cand_T, graphs  host [M], 1 <= M <= SPEC_MAX_CANDIDATES. */
int spec_select_round(const int32_t* chosen_T, int M, const int32_t* cand_T, void* const* graphs,
                      int32_t* launched_out, int32_t* status, cudaStream_t stream);

/* spec_pack_rows -- the packed layout of an allocation applied to a
 * full-depth buffer: dst row row_offsets[i] + j = src row i(K+1) + j for
 * j <= n_i (Section 4.2 "Packing and correctness"), rows of row_bytes bytes.
 * Stands in for a target forward that writes its outputs in packed order.
 *   src             device [B(K+1), row_bytes]; dst device [R_dst, row_bytes]
 *                   (R_dst >= row_offsets[B]; rows past it are not written).
 *   row_offsets     device int32 [B+1] from spec_allocate.
 * A row whose offset within its request exceeds K sets SPEC_ERR_BAD_INPUT. */
int spec_pack_rows(const void* src, size_t row_bytes, int B, int K, const int32_t* row_offsets,
                   void* dst, int R_dst, int32_t* status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * spec_profile_stream_pass -- measurement aid.  The next spec_verify call
 * records `before` immediately before and `after` immediately after its
 * vocabulary-streaming kernel, on its stream, then forgets both.  Arguments
 * are cudaEvent_t handles created by the caller (NULL, NULL cancels).
 * Not thread-safe: meant for a single benchmarking thread.
 * ---------------------------------------------------------------------- */
int spec_profile_stream_pass(cudaEvent_t before, cudaEvent_t after);

/* ------------------------------------------------------------------------
 * spec_check_bounded_wait -- failure-detection check of the library's
 * bounded device waits (the mbarrier waits of spec_markov_draft's
 * tensor-core pipeline).  Launches one warp that waits on an mbarrier no
 * one arrives at: the wait gives up after about a second, sets
 * SPEC_ERR_TIMEOUT in *status (first error wins) and the kernel returns, so
 * the context stays usable.
 *   status          device int32 [1].
 * Returns SPEC_ERR_INVALID_ARG for a NULL status, SPEC_ERR_CUDA if the
 * launch fails, else SPEC_OK (the timeout arrives through *status).
 * ---------------------------------------------------------------------- */
int spec_check_bounded_wait(int32_t* status, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SPEC_H_ */
