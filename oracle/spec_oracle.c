/*
 * spec_oracle.c -- CPU oracle for batched speculative verification.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is a plain, slow, obviously correct
 * restatement of what the GPU path computes, in double precision, one loop per
 * definition.  Only the tests, the smoke check and the benchmark's CPU-baseline
 * leg may load it; the product path never does.  It shares no code, header or
 * constant table with the CUDA library.
 *
 * What it follows (arxiv 2607.25852, "AngelSpec"):
 *   - Section 1: a drafter proposes tokens, the target verifies them in one pass
 *     with rejection sampling, and the verified prefix plus one target token is
 *     committed without changing the target distribution.
 *   - Section 2, Eq. (mtp-acceptance-tv): single-position acceptance under
 *     rejection sampling is sum_v min(p(v), q(v)).
 *   - Section 4.2, Eqs. (dcut-score), (dcut-expected-advance), (dcut-budget),
 *     (dcut-batch-utility), (dcut-select): prefix-survival scores, global top-T
 *     selection with ties toward shallower positions, utility over candidate
 *     budgets and the runtime argmax of utility / cost; "Packing and
 *     correctness" paragraph: dense packing of the unequal prefixes, and the
 *     deterministic-draft, target-only protocol (one-hot q).
 *
 * Readings where the paper is silent:
 *   - verification rule: standard speculative sampling (accept draft z with
 *     probability min(1, p(z)/q(z)); on the first rejection draw from
 *     norm(max(0, p - q)); if every draft is accepted draw the bonus from p);
 *   - row j of a request verifies draft z_{j+1}; the bonus row is row n;
 *   - accept iff u < r with u in [0,1);
 *   - uniforms come from Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11)
 *     with the counter layout below; the draw from a weight vector w is a
 *     two-level exponential race: entries are grouped in blocks of 256
 *     consecutive indices with block weights W_b = sum_{v in b} w_v; the block
 *     b* = argmin_{W_b > 0} E_b / W_b is drawn first, then the entry
 *     y = argmin_{v in b*, w_v > 0} E'_v / w_v (ties to the lowest index at
 *     both levels).  Each level is an exact draw (P(b*) = W_b / W,
 *     P(y | b*) = w_y / W_b), so P(y) = w_y / W.  Every draw (verification,
 *     the drafter's step and the Markov head's step) uses these 256-entry
 *     blocks: an exact draw is all the method asks for, and a draw costs
 *     V / 256 + 256 variates, near the minimum 2 sqrt(V) of V / b + b for the
 *     vocabularies of 128K-201K entries the method serves;
 *   - temperature 0 is the longest argmax-matching prefix plus the argmax of
 *     the first unmatched row (ties to lowest index);
 *   - allocator scores are fp32 products taken in order k = 1..K (the
 *     precision that decides the integer depths on the device too); utility is
 *     the exact integer sum of floor(s * 2^40); the chosen budget is the first
 *     maximiser of utility / cost in candidate order.
 *
 * Counter layout (frozen): key = (lo32(seed), hi32(seed));
 *   counter = (lo32(position), lo32(request), hi32(request), purpose<<28 | sub)
 *   purpose ACCEPT = 1 (sub = 0, word 0 used), SAMPLE = 2 (block variates:
 *   sub = b / 4, word b % 4), SAMPLE_IN_BLOCK = 3 (entry variates: sub = v / 4,
 *   word v % 4); the drafter's draw uses DRAFT = 4 and DRAFT_IN_BLOCK = 5 in
 *   the same way.  Acceptance uniform: (x >> 8) * 2^-24.  Race variate:
 *   E = -ln((2 * (x >> 9) + 1) * 2^-24), the midpoint of one of 2^23 equal
 *   cells of (0, 1), so that E > 0: a variate of exactly 0 would make its entry
 *   win whatever its weight, and the draw would no longer follow w / sum(w).
 *
 * Build: gcc -O2 -ffp-contract=off -fPIC -shared (see oracle/build.py).
 * -ffp-contract=off keeps results identical on x86-64 and aarch64.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_ERR_INVALID_ARG 1
#define OR_ERR_BAD_INPUT 4

#define OR_BF16 0
#define OR_F32 1

#define OR_MODE_GREEDY 0
#define OR_MODE_RESIDUAL 1
#define OR_MODE_BONUS 2
#define OR_MODE_RESIDUAL_EMPTY 3 /* residual mass was zero: drew from p */

#define OR_PURPOSE_ACCEPT 1u
#define OR_PURPOSE_SAMPLE 2u
#define OR_PURPOSE_SAMPLE_IN_BLOCK 3u
#define OR_PURPOSE_DRAFT 4u          /* the drafter's draw: block variates */
#define OR_PURPOSE_DRAFT_IN_BLOCK 5u /* the drafter's draw: entry variates */
#define OR_RACE_BLOCK 256 /* entries per level-1 block, the same for every draw */

/* ------------------------------------------------------------------------ */
/* Element access.  bf16 is the upper half of an IEEE binary32 word.        */
/* ------------------------------------------------------------------------ */
static double load_value(const void* base, int dtype, int64_t idx) {
  if (dtype == OR_F32) {
    return (double)((const float*)base)[idx];
  }
  uint32_t bits = ((uint32_t)((const uint16_t*)base)[idx]) << 16;
  float f;
  memcpy(&f, &bits, sizeof f);
  return (double)f;
}

/* ------------------------------------------------------------------------ */
/* Philox4x32-10 (Salmon et al., SC'11, "Parallel random numbers: as easy   */
/* as 1, 2, 3").  Each round multiplies counter words 0 and 2 by the two    */
/* round multipliers, swaps and XORs the high halves with the round key;    */
/* the key is bumped by the two Weyl constants between rounds.              */
/* ------------------------------------------------------------------------ */
void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2],
                          uint32_t out[4]) {
  const uint32_t mult0 = 0xD2511F53u, mult1 = 0xCD9E8D57u;
  const uint32_t weyl0 = 0x9E3779B9u, weyl1 = 0xBB67AE85u;
  uint32_t x[4] = {ctr[0], ctr[1], ctr[2], ctr[3]};
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += weyl0;
      k1 += weyl1;
    }
    uint64_t prod0 = (uint64_t)mult0 * (uint64_t)x[0];
    uint64_t prod1 = (uint64_t)mult1 * (uint64_t)x[2];
    uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
    uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
    uint32_t y0 = hi1 ^ x[1] ^ k0;
    uint32_t y1 = lo1;
    uint32_t y2 = hi0 ^ x[3] ^ k1;
    uint32_t y3 = lo0;
    x[0] = y0;
    x[1] = y1;
    x[2] = y2;
    x[3] = y3;
  }
  out[0] = x[0];
  out[1] = x[1];
  out[2] = x[2];
  out[3] = x[3];
}

static void draw_words(uint64_t seed, uint64_t request, uint64_t position,
                       uint32_t purpose, uint32_t sub, uint32_t out[4]) {
  uint32_t ctr[4] = {(uint32_t)position, (uint32_t)request,
                     (uint32_t)(request >> 32), (purpose << 28) | sub};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  oracle_philox4x32_10(ctr, key, out);
}

/* Acceptance uniform u in [0, 1) for the draft verified at `position`. */
double oracle_accept_uniform(uint64_t seed, uint64_t request,
                             uint64_t position) {
  uint32_t w[4];
  draw_words(seed, request, position, OR_PURPOSE_ACCEPT, 0u, w);
  return (double)(w[0] >> 8) * ldexp(1.0, -24);
}

/* Unit exponential variate of one Philox word: the word's top 23 bits pick a
 * cell of (0, 1) and u is that cell's midpoint, so 0 < u < 1 and E > 0. */
double oracle_race_variate(uint32_t word) {
  double u = (double)(2u * (word >> 9) + 1u) * ldexp(1.0, -24);
  return -log(u);
}

/* Exponential variate number `index` of purpose `purpose` at `position`:
 * word index % 4 of the Philox call with sub-index index / 4. */
static double race_exponential_with(uint64_t seed, uint64_t request,
                                    uint64_t position, uint32_t purpose,
                                    uint32_t index) {
  uint32_t w[4];
  draw_words(seed, request, position, purpose, index >> 2, w);
  return oracle_race_variate(w[index & 3u]);
}

/* Exponential variate of the sampling race at `position`: level 1 (block b,
 * level = 1) or level 2 (entry v, level = 2). */
double oracle_race_exponential(uint64_t seed, uint64_t request,
                               uint64_t position, uint32_t index, int level) {
  return race_exponential_with(seed, request, position,
                               level == 1 ? OR_PURPOSE_SAMPLE : OR_PURPOSE_SAMPLE_IN_BLOCK,
                               index);
}

/* Two-level exponential race over weights w[0..V) (see the file header),
 * with block variates of purpose `pb` and entry variates of purpose `pe`.
 * race_out[9]: best block key, best block, second block key, second block,
 * the winner y in the best block, its key, the second key in that block, the
 * second entry in that block, and the winner in the second block (-1 if
 * none).  Returns y, or -1 if every weight is zero. */
static int two_level_race_with(const double* w, int V, uint64_t seed,
                               uint64_t request, uint64_t position,
                               uint32_t pb, uint32_t pe, int block,
                               double* race_out) {
  const int nb = (V + block - 1) / block;
  double b1k = INFINITY, b2k = INFINITY;
  int b1 = -1, b2 = -1;
  for (int b = 0; b < nb; ++b) {
    double W = 0.0;
    for (int v = b * block; v < V && v < (b + 1) * block; ++v)
      W += w[v];
    if (!(W > 0.0)) continue;
    double key = race_exponential_with(seed, request, position, pb, (uint32_t)b) / W;
    if (key < b1k) {
      b2k = b1k;
      b2 = b1;
      b1k = key;
      b1 = b;
    } else if (key < b2k) {
      b2k = key;
      b2 = b;
    }
  }
  double yk[2] = {INFINITY, INFINITY}, y2k = INFINITY;
  int y[2] = {-1, -1}, y2 = -1;
  for (int pass = 0; pass < 2; ++pass) {
    int b = pass == 0 ? b1 : b2;
    if (b < 0) continue;
    for (int v = b * block; v < V && v < (b + 1) * block; ++v) {
      if (!(w[v] > 0.0)) continue;
      double key = race_exponential_with(seed, request, position, pe, (uint32_t)v) / w[v];
      if (key < yk[pass]) {
        if (pass == 0) {
          y2k = yk[0];
          y2 = y[0];
        }
        yk[pass] = key;
        y[pass] = v;
      } else if (pass == 0 && key < y2k) {
        y2k = key;
        y2 = v;
      }
    }
  }
  if (race_out) {
    race_out[0] = b1k;
    race_out[1] = b1;
    race_out[2] = b2k;
    race_out[3] = b2;
    race_out[4] = y[0];
    race_out[5] = yk[0];
    race_out[6] = y2k;
    race_out[7] = y2;
    race_out[8] = y[1];
  }
  return y[0];
}

/* The verification draw (purposes SAMPLE and SAMPLE_IN_BLOCK). */
static int two_level_race(const double* w, int V, uint64_t seed,
                          uint64_t request, uint64_t position,
                          double* race_out) {
  return two_level_race_with(w, V, seed, request, position, OR_PURPOSE_SAMPLE,
                             OR_PURPOSE_SAMPLE_IN_BLOCK, OR_RACE_BLOCK, race_out);
}

/* ------------------------------------------------------------------------ */
/* Softmax at temperature t of one row: m = max_v l_v / t,                  */
/* S = sum_v exp(l_v / t - m).  Returns 0 when the row is unusable (a NaN,  */
/* a +inf, or no finite entry).                                             */
/* ------------------------------------------------------------------------ */
static int row_softmax_stats(const void* row, int dtype, int V, double t,
                             double* m_out, double* S_out) {
  double m = -INFINITY;
  for (int v = 0; v < V; ++v) {
    double l = load_value(row, dtype, v);
    if (isnan(l) || l == INFINITY) return 0;
    double x = l / t;
    if (x > m) m = x;
  }
  if (m == -INFINITY) return 0;
  double S = 0.0;
  for (int v = 0; v < V; ++v) {
    double x = load_value(row, dtype, v) / t;
    S += exp(x - m);
  }
  *m_out = m;
  *S_out = S;
  return 1;
}

/* Target probability p(v) of a row with statistics (m, S). */
static double row_prob(const void* row, int dtype, int v, double t, double m,
                       double S) {
  return exp(load_value(row, dtype, v) / t - m) / S;
}

/* Argmax of a row, lowest index on ties; -1 if the row holds a NaN. */
static int row_argmax(const void* row, int dtype, int V, double* max_out) {
  int best = -1;
  double best_val = -INFINITY;
  for (int v = 0; v < V; ++v) {
    double l = load_value(row, dtype, v);
    if (isnan(l)) return -1;
    if (best < 0 || l > best_val) {
      best = v;
      best_val = l;
    }
  }
  *max_out = best_val;
  return best;
}

void oracle_row_stats(const void* row, int dtype, int V, double t,
                      double* m_out, double* S_out, int32_t* ok_out) {
  *ok_out = row_softmax_stats(row, dtype, V, t, m_out, S_out);
}

/* ------------------------------------------------------------------------ */
/* Verification of one request.                                             */
/*   logits  : rows 0..n of this request, row-major [n+1, V]                */
/*   drafts  : z_1..z_n                                                     */
/*   q       : draft distributions of rows 0..n-1 [n, V], or NULL = one-hot */
/*             at the draft token (deterministic-draft protocol)            */
/* Outputs (any pointer may be NULL except accepted/tokens):                */
/*   accepted_out   : a = number of accepted drafts                         */
/*   tokens_out[n+1]: z_1..z_a, y, then -1                                  */
/*   p_draft_out[n] : p_j(z_{j+1})                                          */
/*   row_m_out, row_logS_out [n+1] : m_j and ln S_j (t > 0); max l and 0    */
/*   u_out, r_out [n] : acceptance uniform and ratio per draft (t > 0)      */
/*   race_out[9]    : the two-level race record (two_level_race)             */
/*   mode_out       : OR_MODE_*                                             */
/* Returns OR_OK, or OR_ERR_BAD_INPUT (then a = 0 and tokens[0] = -1).      */
/* ------------------------------------------------------------------------ */
int oracle_verify_request(const void* logits, int logits_dtype,
                          const int32_t* drafts, const void* q, int q_dtype,
                          int n, int V, double t, uint64_t seed,
                          uint64_t request, int64_t pos_base,
                          int32_t* accepted_out, int32_t* tokens_out,
                          double* p_draft_out, double* row_m_out,
                          double* row_logS_out, double* u_out, double* r_out,
                          double* race_out, int32_t* mode_out) {
  for (int j = 0; j <= n; ++j) tokens_out[j] = -1;
  *accepted_out = 0;
  if (race_out) {
    for (int k = 0; k < 9; ++k) race_out[k] = (k == 0 || k == 2 || k == 5 || k == 6) ? INFINITY : -1;
  }
  if (mode_out) *mode_out = t == 0.0 ? OR_MODE_GREEDY : OR_MODE_BONUS;

  int bad = 0;
  if (pos_base < 0 || pos_base + n > (int64_t)0xFFFFFFFF) bad = 1;
  for (int j = 0; j < n; ++j)
    if (drafts[j] < 0 || drafts[j] >= V) bad = 1;

  const size_t esize = logits_dtype == OR_F32 ? 4 : 2;
  const size_t qsize = q_dtype == OR_F32 ? 4 : 2;
#define ROW(j) ((const char*)logits + (size_t)(j) * (size_t)V * esize)
#define QROW(j) ((const char*)q + (size_t)(j) * (size_t)V * qsize)

  if (bad) return OR_ERR_BAD_INPUT;

  /* ---------------- temperature 0: longest argmax-matching prefix ------- */
  if (t == 0.0) {
    int a = 0;
    int matching = 1;
    int y = -1;
    for (int j = 0; j <= n; ++j) {
      double mx;
      int g = row_argmax(ROW(j), logits_dtype, V, &mx);
      if (g < 0) return OR_ERR_BAD_INPUT;
      if (row_m_out) row_m_out[j] = mx;
      if (row_logS_out) row_logS_out[j] = 0.0;
      if (j < n && p_draft_out) p_draft_out[j] = drafts[j] == g ? 1.0 : 0.0;
      if (matching) {
        if (j < n && drafts[j] == g) {
          a = j + 1;
        } else {
          matching = 0;
          y = g;
        }
      }
    }
    for (int j = 0; j < a; ++j) tokens_out[j] = drafts[j];
    tokens_out[a] = y;
    *accepted_out = a;
    return OR_OK;
  }

  /* ---------------- temperature t > 0: rejection sampling --------------- */
  double* m = (double*)malloc(sizeof(double) * (size_t)(n + 1));
  double* S = (double*)malloc(sizeof(double) * (size_t)(n + 1));
  double* w = (double*)malloc(sizeof(double) * (size_t)V);
  int status = OR_OK;
  for (int j = 0; j <= n; ++j) {
    if (!row_softmax_stats(ROW(j), logits_dtype, V, t, &m[j], &S[j])) {
      status = OR_ERR_BAD_INPUT;
      goto done;
    }
    if (row_m_out) row_m_out[j] = m[j];
    if (row_logS_out) row_logS_out[j] = log(S[j]);
  }

  /* Acceptance test of every kept draft; the chain stops at the first
   * rejection (later drafts are reported but do not matter). */
  int a = n;
  int rejected = 0;
  for (int j = 0; j < n; ++j) {
    int z = drafts[j];
    double pz = row_prob(ROW(j), logits_dtype, z, t, m[j], S[j]);
    double qz = q ? load_value(QROW(j), q_dtype, z) : 1.0;
    if (isnan(qz) || qz < 0.0) {
      status = OR_ERR_BAD_INPUT;
      goto done;
    }
    double r;
    if (qz > 0.0)
      r = fmin(1.0, pz / qz);
    else
      r = pz > 0.0 ? 1.0 : 0.0;
    double u = oracle_accept_uniform(seed, request, (uint64_t)(pos_base + j));
    if (p_draft_out) p_draft_out[j] = pz;
    if (u_out) u_out[j] = u;
    if (r_out) r_out[j] = r;
    if (!rejected && !(u < r)) {
      a = j;
      rejected = 1;
    }
  }

  /* Weights of the final draw: residual max(0, p - q) at the rejected row,
   * or p at the bonus row n. */
  int row = a;
  int mode = rejected ? OR_MODE_RESIDUAL : OR_MODE_BONUS;
  double mass = 0.0;
  for (int v = 0; v < V; ++v) {
    double p = row_prob(ROW(row), logits_dtype, v, t, m[row], S[row]);
    if (rejected) {
      double qv = q ? load_value(QROW(row), q_dtype, v)
                    : (v == drafts[row] ? 1.0 : 0.0);
      w[v] = fmax(0.0, p - qv);
    } else {
      w[v] = p;
    }
    mass += w[v];
  }
  if (rejected && mass == 0.0) {
    mode = OR_MODE_RESIDUAL_EMPTY;
    for (int v = 0; v < V; ++v)
      w[v] = row_prob(ROW(row), logits_dtype, v, t, m[row], S[row]);
  }

  /* Two-level exponential race over w at the sampled position. */
  const uint64_t position = (uint64_t)(pos_base + row);
  int best_v = two_level_race(w, V, seed, request, position, race_out);
  if (best_v < 0) {
    status = OR_ERR_BAD_INPUT;
    goto done;
  }
  for (int j = 0; j < a; ++j) tokens_out[j] = drafts[j];
  tokens_out[a] = best_v;
  *accepted_out = a;
  if (mode_out) *mode_out = mode;

done:
  if (status != OR_OK) {
    for (int j = 0; j <= n; ++j) tokens_out[j] = -1;
    *accepted_out = 0;
  }
  free(m);
  free(S);
  free(w);
#undef ROW
#undef QROW
  return status;
}

/* ------------------------------------------------------------------------ */
/* Batched verification, a loop over requests with the same layout as the  */
/* device entry point: logits rows of request i start at row_offsets[i]     */
/* (NULL: i*(K+1)); depth NULL means every request keeps K drafts; q is     */
/* [B, K, V] or NULL.  Per-request outputs are strided by K (p_draft, u, r) */
/* and K+1 (tokens); row statistics are indexed by packed row.              */
/* Returns the first non-OK status seen (every request is still processed). */
/* ------------------------------------------------------------------------ */
int oracle_verify_batch(const void* logits, int logits_dtype,
                        const int32_t* row_offsets, const int32_t* depth,
                        const int32_t* drafts, const void* q, int q_dtype,
                        int B, int K, int V, double t, const uint64_t* seeds,
                        const uint64_t* request_ids, const int64_t* pos_base,
                        int32_t* accepted_out, int32_t* tokens_out,
                        double* p_draft_out, double* row_m_out,
                        double* row_logS_out, double* u_out, double* r_out,
                        double* race_out, int32_t* mode_out,
                        int32_t* status_out) {
  const size_t esize = logits_dtype == OR_F32 ? 4 : 2;
  const size_t qsize = q_dtype == OR_F32 ? 4 : 2;
  int first = OR_OK;
  for (int i = 0; i < B; ++i) {
    int n = depth ? depth[i] : K;
    int64_t row0 = row_offsets ? row_offsets[i] : (int64_t)i * (K + 1);
    int32_t* tok = tokens_out + (size_t)i * (K + 1);
    for (int j = 0; j <= K; ++j) tok[j] = -1;
    int st;
    if (n < 0 || n > K ||
        (row_offsets && row_offsets[i + 1] != row_offsets[i] + n + 1)) {
      accepted_out[i] = 0;
      st = OR_ERR_BAD_INPUT;
    } else {
      st = oracle_verify_request(
          (const char*)logits + (size_t)row0 * (size_t)V * esize,
          logits_dtype, drafts + (size_t)i * K,
          q ? (const void*)((const char*)q + (size_t)i * K * (size_t)V * qsize)
            : NULL,
          q_dtype, n, V, t, seeds[i], request_ids[i], pos_base[i],
          &accepted_out[i], tok,
          p_draft_out ? p_draft_out + (size_t)i * K : NULL,
          row_m_out ? row_m_out + row0 : NULL,
          row_logS_out ? row_logS_out + row0 : NULL,
          u_out ? u_out + (size_t)i * K : NULL,
          r_out ? r_out + (size_t)i * K : NULL,
          race_out ? race_out + (size_t)i * 9 : NULL,
          mode_out ? mode_out + i : NULL);
    }
    if (status_out) status_out[i] = st;
    if (st != OR_OK && first == OR_OK) first = st;
  }
  return first;
}

/* ------------------------------------------------------------------------ */
/* The drafter's producer step (Section 4.2: D-cut reads the drafter's      */
/* token-level confidences c_{i,t}, Eq. dcut-score; the paper does not      */
/* define c further).  Reading: for k = 0..K-1, row k of the drafter's      */
/* logits gives q_k = softmax(l_k / tau), the draft z_{k+1} is drawn from   */
/* q_k by the two-level race at position pos_base + k + 1 (purposes DRAFT   */
/* and DRAFT_IN_BLOCK), or is argmax_v l_k (lowest index) when tau == 0,    */
/* and its confidence is c_{k+1} = q_k(z_{k+1}), with q_k at temperature 1  */
/* when tau == 0.  Scores as the allocator forms them (Eq. dcut-score):     */
/* s_0 = 1, s_k = fl32(s_{k-1} * fl32(c_k)).                                */
/*   logits [K, V] of dtype; z_out [K]; c_out [K] (fp64); s_out [K+1];      */
/*   m_out, logS_out [K]: each row's max_v l_v / tau' and                   */
/*   ln sum_v exp(l_v / tau' - m) (tau' = tau, or 1 when tau == 0);         */
/*   race_out [K][9] or NULL: each row's race record (two_level_race).      */
/* A row with a NaN, a +inf or no finite entry, or a position past 2^32 - 1 */
/* makes the request bad: z = -1, c = 0, s_0 = 1 and s_k = 0 for k >= 1.   */
/* Returns OR_OK or OR_ERR_BAD_INPUT.                                       */
/* ------------------------------------------------------------------------ */
int oracle_draft_request(const void* logits, int dtype, int K, int V, double tau,
                         uint64_t seed, uint64_t request, int64_t pos_base,
                         int32_t* z_out, double* c_out, float* s_out,
                         double* m_out, double* logS_out, double* race_out) {
  const size_t esize = dtype == OR_F32 ? 4 : 2;
  const double tc = tau > 0.0 ? tau : 1.0;
  int bad = pos_base < 0 || pos_base + K > (int64_t)0xFFFFFFFF;
  double* w = (double*)malloc(sizeof(double) * (size_t)(V > 0 ? V : 1));
  s_out[0] = 1.0f;
  for (int k = 0; k < K && !bad; ++k) {
    const void* row = (const char*)logits + (size_t)k * (size_t)V * esize;
    double m, S;
    if (!row_softmax_stats(row, dtype, V, tc, &m, &S)) {
      bad = 1;
      break;
    }
    int z;
    if (tau == 0.0) {
      double mx;
      z = row_argmax(row, dtype, V, &mx);
      if (race_out)
        for (int e = 0; e < 9; ++e) race_out[(size_t)k * 9 + e] = -1;
    } else {
      for (int v = 0; v < V; ++v) w[v] = row_prob(row, dtype, v, tc, m, S);
      z = two_level_race_with(w, V, seed, request, (uint64_t)(pos_base + k + 1), OR_PURPOSE_DRAFT,
                              OR_PURPOSE_DRAFT_IN_BLOCK, OR_RACE_BLOCK, race_out ? race_out + (size_t)k * 9 : NULL);
    }
    if (z < 0) {
      bad = 1;
      break;
    }
    z_out[k] = z;
    c_out[k] = row_prob(row, dtype, z, tc, m, S);
    s_out[k + 1] = s_out[k] * (float)c_out[k];
    m_out[k] = m;
    logS_out[k] = log(S);
  }
  free(w);
  if (bad) {
    for (int k = 0; k < K; ++k) {
      z_out[k] = -1;
      c_out[k] = 0.0;
      s_out[k + 1] = 0.0f;
      m_out[k] = 0.0;
      logS_out[k] = 0.0;
    }
    return OR_ERR_BAD_INPUT;
  }
  return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* The Markov head's sequential draw (Section 3.2, Eq. dspark-markov, after   */
/* the block factorisation Eq. ar-factorization): the drafter's base logits  */
/* U_k of each position get the first-order bias b_k = W1[x_{k-1}] W2 of the */
/* previously drawn token (x_0 the last committed token), and               */
/* q_k = softmax((U_k + b_k) / tau').  Draws, confidences, scores and the    */
/* bad-input rule as in oracle_draft_request, position by position: the     */
/* same two-level race (blocks of OR_RACE_BLOCK entries, purposes DRAFT and  */
/* DRAFT_IN_BLOCK), so that with W1 = 0 the draw is the draft step's.        */
/*   U [K, V] of dtype; W1 [V, r] and W2 [r, V] bf16 bits (uint16).          */
/* ------------------------------------------------------------------------ */
static double bf16_value(uint16_t h) {
  uint32_t w = (uint32_t)h << 16;
  float f;
  memcpy(&f, &w, 4);
  return (double)f;
}

int oracle_markov_request(const void* U, int dtype, const uint16_t* W1, const uint16_t* W2, int K, int V,
                          int r, int32_t x0, double tau, uint64_t seed, uint64_t request,
                          int64_t pos_base, int32_t* z_out, double* c_out, float* s_out,
                          double* m_out, double* logS_out, double* race_out) {
  const size_t esize = dtype == OR_F32 ? 4 : 2;
  const double tc = tau > 0.0 ? tau : 1.0;
  int bad = pos_base < 0 || pos_base + K > (int64_t)0xFFFFFFFF || x0 < 0 || x0 >= V;
  double* l = (double*)malloc(sizeof(double) * (size_t)V);
  double* w = (double*)malloc(sizeof(double) * (size_t)V);
  s_out[0] = 1.0f;
  int prev = x0;
  for (int k = 0; k < K && !bad; ++k) {
    const void* urow = (const char*)U + (size_t)k * (size_t)V * esize;
    /* l = U_k + W1[prev] W2, in double */
    for (int v = 0; v < V; ++v) {
      double b = 0.0;
      for (int j = 0; j < r; ++j) b += bf16_value(W1[(size_t)prev * r + j]) * bf16_value(W2[(size_t)j * V + v]);
      l[v] = load_value(urow, dtype, v) + b;
      if (isnan(l[v]) || l[v] == INFINITY) bad = 1;
    }
    if (bad) break;
    double m = -INFINITY;
    for (int v = 0; v < V; ++v)
      if (l[v] / tc > m) m = l[v] / tc;
    if (m == -INFINITY) {
      bad = 1;
      break;
    }
    double S = 0.0;
    for (int v = 0; v < V; ++v) S += exp(l[v] / tc - m);
    int z = -1;
    if (tau == 0.0) {
      double best = -INFINITY;
      for (int v = 0; v < V; ++v)
        if (z < 0 || l[v] > best) {
          z = v;
          best = l[v];
        }
      if (race_out)
        for (int e = 0; e < 9; ++e) race_out[(size_t)k * 9 + e] = -1;
    } else {
      for (int v = 0; v < V; ++v) w[v] = exp(l[v] / tc - m) / S;
      z = two_level_race_with(w, V, seed, request, (uint64_t)(pos_base + k + 1), OR_PURPOSE_DRAFT,
                              OR_PURPOSE_DRAFT_IN_BLOCK, OR_RACE_BLOCK, race_out ? race_out + (size_t)k * 9 : NULL);
    }
    if (z < 0) {
      bad = 1;
      break;
    }
    z_out[k] = z;
    c_out[k] = exp(l[z] / tc - m) / S;
    s_out[k + 1] = s_out[k] * (float)c_out[k];
    m_out[k] = m;
    logS_out[k] = log(S);
    prev = z;
  }
  free(l);
  free(w);
  if (bad) {
    for (int k = 0; k < K; ++k) {
      z_out[k] = -1;
      c_out[k] = 0.0;
      s_out[k + 1] = 0.0f;
      m_out[k] = 0.0;
      logS_out[k] = 0.0;
    }
    return OR_ERR_BAD_INPUT;
  }
  return OR_OK;
}

/* The drafter's step for B requests: logits [B, K, V]; outputs per request  */
/* as in oracle_draft_request (z [B, K], c [B, K], s [B, K+1], m and logS    */
/* [B, K], race [B, K, 9] or NULL, status [B]).  Returns the first non-OK.   */
int oracle_draft_batch(const void* logits, int dtype, int B, int K, int V, double tau,
                       const uint64_t* seeds, const uint64_t* request_ids,
                       const int64_t* pos_base, int32_t* z_out, double* c_out,
                       float* s_out, double* m_out, double* logS_out,
                       double* race_out, int32_t* status_out) {
  const size_t esize = dtype == OR_F32 ? 4 : 2;
  int first = OR_OK;
  for (int i = 0; i < B; ++i) {
    const size_t r0 = (size_t)i * K;
    int st = oracle_draft_request((const char*)logits + r0 * (size_t)V * esize, dtype, K, V, tau,
                                  seeds[i], request_ids[i], pos_base[i], z_out + r0, c_out + r0,
                                  s_out + (size_t)i * (K + 1), m_out + r0, logS_out + r0,
                                  race_out ? race_out + r0 * 9 : NULL);
    if (status_out) status_out[i] = st;
    if (st != OR_OK && first == OR_OK) first = st;
  }
  return first;
}

/* ------------------------------------------------------------------------ */
/* D-cut allocation (Section 4.2).                                          */
/* ------------------------------------------------------------------------ */
typedef struct {
  float s;
  int k;
  int i;
} position_t;

/* Global order: score descending, then shallower k, then lower request. */
static int position_cmp(const void* pa, const void* pb) {
  const position_t* a = (const position_t*)pa;
  const position_t* b = (const position_t*)pb;
  if (a->s != b->s) return a->s > b->s ? -1 : 1;
  if (a->k != b->k) return a->k < b->k ? -1 : 1;
  if (a->i != b->i) return a->i < b->i ? -1 : 1;
  return 0;
}

/* Q(s) = floor(s * 2^40): the fixed-point utility of one kept position. */
static int64_t utility_units(float s) {
  return (int64_t)floor(ldexp((double)s, 40));
}

/* Eq. (dcut-budget) in exact integers: max(B, ceil(num/den * B(K+1))). */
int oracle_budget(int B, int K, int64_t num, int64_t den) {
  int64_t full = (int64_t)B * (K + 1);
  int64_t T = (num * full + den - 1) / den;
  if (T < B) T = B;
  return (int)T;
}

/*
 * conf [B, K] fp32: c_{i,t} for t = 1..K.  cand_T [M] budgets (each in
 * [B, B(K+1)]), cand_cost [M] > 0.  Outputs: depth [B] (n_i at the chosen
 * budget), row_offsets [B+1], packed tokens / positions [B(K+1)] (row 0 of a
 * request carries its last committed token, row j the draft z_j; unused rows
 * are -1), chosen_T, utility [M] in token units, all_depths [M, B] (optional).
 * An invalid confidence (NaN or outside [0, 1]) counts as 0 and yields
 * OR_ERR_BAD_INPUT.
 */
int oracle_allocate(const float* conf, int B, int K, const int32_t* cand_T,
                    const double* cand_cost, int M, const int32_t* last_tokens,
                    const int32_t* drafts, const int64_t* pos_base,
                    int32_t* depth_out, int32_t* row_offsets_out,
                    int32_t* packed_tokens_out, int64_t* packed_pos_out,
                    int32_t* chosen_T_out, double* utility_out,
                    int32_t* all_depths_out) {
  if (B <= 0 || K < 0 || M <= 0) return OR_ERR_INVALID_ARG;
  const int N = B * (K + 1);
  for (int c = 0; c < M; ++c) {
    if (cand_T[c] < B || cand_T[c] > N) return OR_ERR_INVALID_ARG;
    if (!(cand_cost[c] > 0.0) || isinf(cand_cost[c])) return OR_ERR_INVALID_ARG;
  }
  int status = OR_OK;

  /* Eq. (dcut-score): s_{i,0} = 1, s_{i,k} = prod_{t<=k} c_{i,t} (fp32, in order). */
  float* s = (float*)malloc(sizeof(float) * (size_t)N);
  for (int i = 0; i < B; ++i) {
    float acc = 1.0f;
    s[i * (K + 1)] = acc;
    for (int k = 1; k <= K; ++k) {
      float c = conf[(size_t)i * K + (k - 1)];
      if (!(c >= 0.0f && c <= 1.0f)) {
        status = OR_ERR_BAD_INPUT;
        c = 0.0f;
      }
      acc = acc * c;
      s[i * (K + 1) + k] = acc;
    }
  }

  /* Global ranking of all B(K+1) positions. */
  position_t* order = (position_t*)malloc(sizeof(position_t) * (size_t)N);
  for (int i = 0; i < B; ++i)
    for (int k = 0; k <= K; ++k) {
      order[i * (K + 1) + k].s = s[i * (K + 1) + k];
      order[i * (K + 1) + k].k = k;
      order[i * (K + 1) + k].i = i;
    }
  qsort(order, (size_t)N, sizeof(position_t), position_cmp);

  /* For each candidate budget: keep depths from the top-T positions, then
   * Eq. (dcut-batch-utility) U = sum_i sum_{k=0}^{n_i} s_{i,k}. */
  int* kept = (int*)malloc(sizeof(int) * (size_t)B);
  int* depth_c = (int*)malloc(sizeof(int) * (size_t)B * (size_t)M);
  double best_obj = -INFINITY;
  int best_c = 0;
  for (int c = 0; c < M; ++c) {
    for (int i = 0; i < B; ++i) kept[i] = 0;
    for (int p = 0; p < cand_T[c]; ++p) kept[order[p].i] += 1;
    int64_t U = 0;
    for (int i = 0; i < B; ++i) {
      int n = kept[i] - 1;
      depth_c[(size_t)c * B + i] = n;
      for (int k = 0; k <= n; ++k) U += utility_units(s[i * (K + 1) + k]);
    }
    double util = ldexp((double)U, -40);
    if (utility_out) utility_out[c] = util;
    /* Eq. (dcut-select): first maximiser of U / C. */
    double obj = util / cand_cost[c];
    if (obj > best_obj) {
      best_obj = obj;
      best_c = c;
    }
  }
  if (all_depths_out)
    memcpy(all_depths_out, depth_c, sizeof(int32_t) * (size_t)B * (size_t)M);

  /* Dense packing of the chosen prefixes. */
  *chosen_T_out = cand_T[best_c];
  for (int p = 0; p < N; ++p) {
    packed_tokens_out[p] = -1;
    packed_pos_out[p] = -1;
  }
  int32_t off = 0;
  for (int i = 0; i < B; ++i) {
    int n = depth_c[(size_t)best_c * B + i];
    depth_out[i] = n;
    row_offsets_out[i] = off;
    for (int j = 0; j <= n; ++j) {
      packed_tokens_out[off + j] =
          j == 0 ? last_tokens[i] : drafts[(size_t)i * K + (j - 1)];
      packed_pos_out[off + j] = pos_base[i] + j;
    }
    off += n + 1;
  }
  row_offsets_out[B] = off;

  free(s);
  free(order);
  free(kept);
  free(depth_c);
  return status;
}

/* ------------------------------------------------------------------------ */
/* Commit: committed tokens z_1..z_a, y of each request packed back to back */
/* (offsets are the exclusive scan of a_i + 1), and target hidden rows      */
/* 0..a_i of each request gathered in the same order.                       */
/* ------------------------------------------------------------------------ */
void oracle_commit(const int32_t* accepted, const int32_t* tokens,
                   const int32_t* row_offsets, const void* hidden,
                   int64_t row_bytes, int B, int K, int32_t* packed_tokens_out,
                   int32_t* commit_offsets_out, void* hidden_out) {
  int32_t off = 0;
  for (int i = 0; i < B; ++i) {
    int a = accepted[i];
    int64_t row0 = row_offsets ? row_offsets[i] : (int64_t)i * (K + 1);
    commit_offsets_out[i] = off;
    for (int j = 0; j <= a; ++j) {
      packed_tokens_out[off + j] = tokens[(size_t)i * (K + 1) + j];
      if (hidden && hidden_out)
        memcpy((char*)hidden_out + (size_t)(off + j) * (size_t)row_bytes,
               (const char*)hidden + (size_t)(row0 + j) * (size_t)row_bytes,
               (size_t)row_bytes);
    }
    off += a + 1;
  }
  commit_offsets_out[B] = off;
}
