/*
 * dcd_oracle.c -- plain, slow, fp64 CPU oracle of the contrastive-decoding (CD)
 * verification step of Decoupled Contrastive Decoding (arxiv 2608.12913).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test-suite, the smoke check and the
 * benchmark's CPU-baseline leg load this library.  It shares no code, header,
 * table or constant with the CUDA path, and the CUDA path never calls it.
 *
 * What it computes, per row (the next-token logits after one draft-tree node),
 * straight from the paper's definitions, every step in double precision from
 * the exact input values:
 *
 *   1. log pi_p = z_p - logsumexp(z_p), log pi_q = z_q - logsumexp(z_q)
 *      (the two softmax distributions of Sec. 2.1);
 *   2. plausibility set P_beta = {x : pi_p(x) >= beta * max pi_p} (Sec. 2.1),
 *      the whole vocabulary when beta = 0 (the paper's "untruncated target");
 *   3. log-form CD score (1+alpha) log pi_p - alpha log pi_q on P_beta (Eq. 1);
 *   4. pi_CD,T proportional to exp(score / T) on P_beta, zero off it; T = 0
 *      (greedy) uses the argmax of the score and T = 1 for reported log-probs;
 *   5. greedy rule (T = 0): a child is accepted iff its token is the argmax of
 *      its parent's row (the T -> 0 limit of Algorithm 1);
 *   6. sampled rule (T > 0), Algorithm 1 generalised to sibling lists: with
 *      r_0 = pi_CD, child j (ascending node id) is accepted iff
 *      u_j <= r_{j-1}(t_j) / q(t_j); on rejection r_j = normalise(max(0,
 *      r_{j-1} - q)); if no child is accepted, the row's terminal token is drawn
 *      from the last residual (pi_CD itself at a leaf), "sample y_k ~ P_r".
 *      With siblings drawn without replacement ("distinct"), sibling j's proposal
 *      q_{j-1} is q with the tokens of siblings 1..j-1 removed and renormalised, and it
 *      takes q's place in both the ratio and the residual step;
 *   7. tree walk: from the root, descend into the accepted child while there is
 *      one; accept_len = number of accepted drafted tokens (the bonus token is
 *      excluded, App. D), the bonus is the terminal token of the last node.
 *
 * Randomness (the paper fixes none; this is the library's own convention):
 * Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy
 * as 1, 2, 3", SC'11), key = (seed_lo, seed_hi).  The acceptance uniform of
 * node c (global id G = b*N + c) uses counter (G, 0, off_lo, off_hi), word 0;
 * the race uniform of token x in row G uses counter (G, 1 + x/4, off_lo,
 * off_hi), word x%4; the race uniform of token block k (ids 1024k .. 1024k+1023)
 * uses counter (G, 2^31 + k/4, off_lo, off_hi), word k%4.  A 32-bit word w
 * becomes u = ((w >> 9) + 0.5) * 2^-23, a value in (0, 1) that fp32 also holds
 * exactly.  Terminal tokens are drawn by a two-level exponential race: a block
 * by argmax_k log R_k - log(-log u_k) over the blocks' masses R_k, then a token
 * of that block by argmax_x log r(x) - log(-log u_x); ties to the lowest id.
 *
 * Besides the outputs, every row reports decision margins (top-2 score gap,
 * |u - ratio| of every acceptance test taken, top-2 race-key gap, distance of
 * the nearest logit to the plausibility threshold) so that a test can tell a
 * genuine disagreement from an fp32-versus-fp64 near-tie.
 *
 * Build: gcc -O2 -std=c11 -fPIC -shared [-fopenmp] dcd_oracle.c -lm
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_OK 0
#define ORC_ERR_ARG (-1)
#define ORC_ERR_TREE (-2)
#define ORC_ERR_MEM (-7)

/* ---------------------------------------------------------------- Philox */

static void philox_round(uint32_t c[4], const uint32_t k[2]) {
  const uint64_t p0 = (uint64_t)0xD2511F53u * c[0];
  const uint64_t p1 = (uint64_t)0xCD9E8D57u * c[2];
  const uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
  const uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
  const uint32_t n0 = hi1 ^ c[1] ^ k[0];
  const uint32_t n2 = hi0 ^ c[3] ^ k[1];
  c[0] = n0;
  c[1] = lo1;
  c[2] = n2;
  c[3] = lo0;
}

/* Philox4x32 with 10 rounds; the key is bumped by the Weyl constants between rounds. */
void dcd_oracle_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4]) {
  uint32_t c[4] = {ctr_in[0], ctr_in[1], ctr_in[2], ctr_in[3]};
  uint32_t k[2] = {key_in[0], key_in[1]};
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k[0] += 0x9E3779B9u;
      k[1] += 0xBB67AE85u;
    }
    philox_round(c, k);
  }
  memcpy(out, c, sizeof c);
}

double dcd_oracle_u01(uint32_t w) { return ((double)(w >> 9) + 0.5) * (1.0 / 8388608.0); }

static uint32_t philox_word(uint64_t seed, uint64_t offset, uint32_t w0, uint32_t w1, int word) {
  uint32_t ctr[4] = {w0, w1, (uint32_t)offset, (uint32_t)(offset >> 32)};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t out[4];
  dcd_oracle_philox4x32_10(ctr, key, out);
  return out[word];
}

/* Acceptance uniform of global node id G. */
double dcd_oracle_accept_uniform(uint64_t seed, uint64_t offset, uint32_t G) {
  return dcd_oracle_u01(philox_word(seed, offset, G, 0u, 0));
}

/* Exponential-race uniform of token x in global row G. */
double dcd_oracle_race_uniform(uint64_t seed, uint64_t offset, uint32_t G, int64_t x) {
  return dcd_oracle_u01(philox_word(seed, offset, G, (uint32_t)(1 + (x >> 2)), (int)(x & 3)));
}

/* Exponential-race uniform of token block k (tokens 1024k .. 1024k+1023) in global row G. */
double dcd_oracle_block_uniform(uint64_t seed, uint64_t offset, uint32_t G, int64_t k) {
  return dcd_oracle_u01(philox_word(seed, offset, G, 0x80000000u | (uint32_t)(k >> 2), (int)(k & 3)));
}

/* ---------------------------------------------------------------- inputs */

/* dtype: 0 = fp32, 1 = bf16 (raw 16-bit pattern), 2 = fp64. */
static double logit_at(const void* base, int dtype, int64_t i) {
  if (dtype == 0) return (double)((const float*)base)[i];
  if (dtype == 1) {
    uint32_t bits = (uint32_t)((const uint16_t*)base)[i] << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
  }
  return ((const double*)base)[i];
}

static size_t dtype_size(int dtype) { return dtype == 0 ? 4 : (dtype == 1 ? 2 : 8); }

/* ---------------------------------------------------------------- per-row CD target */

typedef struct {
  double lse_p;      /* logsumexp of the expert logits */
  double lse_q;      /* logsumexp of the amateur logits */
  double log_zcd;    /* log sum_{P_beta} exp(score / T_eff): the paper's log Z_CD at T_eff */
  double cd_lse;     /* log sum_{P_beta} exp(s'(x) / T_eff) with raw s' = (1+a) z_p - a z_q */
  double gap_argmax; /* score(argmax) - score(runner-up) on P_beta (+inf if |P_beta| = 1) */
  double gap_mask;   /* min_x |log pi_p(x) - max log pi_p - log beta| (+inf when beta = 0) */
  int32_t argmax;    /* argmax_{P_beta} score, lowest id on ties */
  int32_t n_mask;    /* |P_beta| */
} orc_row_target;

/*
 * Fills logpi[V] = log pi_CD,T(x) (-inf off the plausibility set) and the row summary.
 * lp/lq are scratch arrays of length V.
 */
static void row_target(int64_t V, int dtype, const void* zp, const void* zq, double alpha, double beta,
                       double T, double* lp, double* lq, double* logpi, orc_row_target* st) {
  const double T_eff = T > 0.0 ? T : 1.0;
  /* step 1: the two log-softmax distributions */
  double mp = -INFINITY, mq = -INFINITY;
  for (int64_t x = 0; x < V; ++x) {
    lp[x] = logit_at(zp, dtype, x);
    lq[x] = logit_at(zq, dtype, x);
    if (lp[x] > mp) mp = lp[x];
    if (lq[x] > mq) mq = lq[x];
  }
  double sp = 0.0, sq = 0.0;
  for (int64_t x = 0; x < V; ++x) {
    sp += exp(lp[x] - mp);
    sq += exp(lq[x] - mq);
  }
  st->lse_p = mp + log(sp);
  st->lse_q = mq + log(sq);
  double max_lp = -INFINITY;
  for (int64_t x = 0; x < V; ++x) {
    lp[x] -= st->lse_p;
    lq[x] -= st->lse_q;
    if (lp[x] > max_lp) max_lp = lp[x];
  }
  /* step 2: plausibility set P_beta = {x : pi_p(x) >= beta * max pi_p} */
  const double log_beta = beta > 0.0 ? log(beta) : -INFINITY;
  st->gap_mask = INFINITY;
  /* steps 3-4: log-form score on P_beta, its argmax and the normaliser */
  double best = -INFINITY, second = -INFINITY, mscore = -INFINITY;
  int32_t arg = -1, nm = 0;
  for (int64_t x = 0; x < V; ++x) {
    int in = 1;
    if (beta > 0.0) {
      const double d = lp[x] - max_lp - log_beta;
      if (fabs(d) < st->gap_mask) st->gap_mask = fabs(d);
      in = d >= 0.0;
    }
    if (!in) {
      logpi[x] = -INFINITY;
      continue;
    }
    ++nm;
    const double score = (1.0 + alpha) * lp[x] - alpha * lq[x];
    logpi[x] = score; /* temporarily the score */
    if (score > best) {
      second = best;
      best = score;
      arg = (int32_t)x;
    } else if (score > second) {
      second = score;
    }
    if (score / T_eff > mscore) mscore = score / T_eff;
  }
  double ssum = 0.0;
  for (int64_t x = 0; x < V; ++x)
    if (logpi[x] > -INFINITY) ssum += exp(logpi[x] / T_eff - mscore);
  st->log_zcd = mscore + log(ssum);
  for (int64_t x = 0; x < V; ++x)
    if (logpi[x] > -INFINITY) logpi[x] = logpi[x] / T_eff - st->log_zcd;
  st->argmax = arg;
  st->n_mask = nm;
  st->gap_argmax = (nm > 1) ? best - second : INFINITY;
  /* the same normaliser in the raw-logit form used by the library's outputs */
  double mraw = -INFINITY;
  for (int64_t x = 0; x < V; ++x)
    if (logpi[x] > -INFINITY) {
      const double s = ((1.0 + alpha) * logit_at(zp, dtype, x) - alpha * logit_at(zq, dtype, x)) / T_eff;
      if (s > mraw) mraw = s;
    }
  double sraw = 0.0;
  for (int64_t x = 0; x < V; ++x)
    if (logpi[x] > -INFINITY) {
      const double s = ((1.0 + alpha) * logit_at(zp, dtype, x) - alpha * logit_at(zq, dtype, x)) / T_eff;
      sraw += exp(s - mraw);
    }
  st->cd_lse = mraw + log(sraw);
}

/* r <- normalise(max(0, r - q)); returns the mass before normalising.  When the mass is
 * zero the residual is left unchanged (then r == q, and rejection cannot happen). */
static double residual_step(int64_t V, double* r, const float* q, double* tmp) {
  double z = 0.0;
  for (int64_t x = 0; x < V; ++x) {
    const double d = r[x] - (double)q[x];
    tmp[x] = d > 0.0 ? d : 0.0;
    z += tmp[x];
  }
  if (z > 0.0)
    for (int64_t x = 0; x < V; ++x) r[x] = tmp[x] / z;
  return z;
}

/* The same step against a proposal held in double precision (the renormalised proposal of a
 * sibling drawn without replacement). */
static double residual_step_d(int64_t V, double* r, const double* qd, double* tmp) {
  double z = 0.0;
  for (int64_t x = 0; x < V; ++x) {
    const double d = r[x] - qd[x];
    tmp[x] = d > 0.0 ? d : 0.0;
    z += tmp[x];
  }
  if (z > 0.0)
    for (int64_t x = 0; x < V; ++x) r[x] = tmp[x] / z;
  return z;
}

/* Siblings drawn without replacement: after sibling token t is rejected, the next sibling's
 * proposal is q with t removed and renormalised.  qd holds the current proposal. */
static void remove_token(int64_t V, double* qd, int32_t t) {
  if (qd[t] == 0.0) return; /* already removed (a duplicate sibling) */
  qd[t] = 0.0;
  double z = 0.0;
  for (int64_t x = 0; x < V; ++x) z += qd[x];
  if (z > 0.0)
    for (int64_t x = 0; x < V; ++x) qd[x] /= z;
}

/* Acceptance ratio r(t)/q(t); q(t) = 0 gives +inf if r(t) > 0 and 0 (reject) otherwise. */
static double accept_ratio(double rt, double qt) {
  if (qt > 0.0) return rt / qt;
  return rt > 0.0 ? INFINITY : 0.0;
}

#define RACE_BLOCK 1024

/*
 * Draw from r (unnormalised, r >= 0) by a two-level exponential race: first a block of
 * RACE_BLOCK consecutive token ids, k* = argmax_k log R_k - log(-log u_k) with R_k the block's
 * mass, then a token of that block, argmax_x log r(x) - log(-log u_x).  Each level is a
 * Gumbel-max draw, so P(x) = (R_k / sum R) (r(x) / R_k) = r(x) / sum r, with k the block of x.
 * Ties go to the lowest id.
 * Writes the smaller of the two levels' top-2 key gaps.
 */
static int32_t race(int64_t V, const double* r, uint64_t seed, uint64_t offset, uint32_t G, double* gap) {
  const int64_t nblk = (V + RACE_BLOCK - 1) / RACE_BLOCK;
  double best = -INFINITY, second = -INFINITY;
  int64_t kbest = -1;
  for (int64_t k = 0; k < nblk; ++k) {
    double mass = 0.0;
    for (int64_t x = k * RACE_BLOCK; x < V && x < (k + 1) * RACE_BLOCK; ++x) mass += r[x];
    if (!(mass > 0.0)) continue;
    const double u = dcd_oracle_block_uniform(seed, offset, G, k);
    const double key = log(mass) - log(-log(u));
    if (key > best) {
      second = best;
      best = key;
      kbest = k;
    } else if (key > second) {
      second = key;
    }
  }
  const double gap1 = best - second;
  best = -INFINITY;
  second = -INFINITY;
  int32_t arg = -1;
  if (kbest >= 0) {
    for (int64_t x = kbest * RACE_BLOCK; x < V && x < (kbest + 1) * RACE_BLOCK; ++x) {
      if (!(r[x] > 0.0)) continue;
      const double u = dcd_oracle_race_uniform(seed, offset, G, x);
      const double key = log(r[x]) - log(-log(u));
      if (key > best) {
        second = best;
        best = key;
        arg = (int32_t)x;
      } else if (key > second) {
        second = key;
      }
    }
  }
  const double gap2 = best - second;
  *gap = gap1 < gap2 ? gap1 : gap2;
  return arg;
}

/* ---------------------------------------------------------------- exported helpers for the pins */

/* log pi_CD,T of one row (T = 0 reports the T = 1 distribution) and its summary. */
int dcd_oracle_row_logpi(int64_t V, int dtype, const void* zp, const void* zq, double alpha, double beta,
                         double T, double* logpi, double* lse_p, double* lse_q, double* log_zcd,
                         double* cd_lse, int32_t* argmax, double* gap_argmax) {
  if (V <= 0 || !zp || !zq || !logpi) return ORC_ERR_ARG;
  double* lp = malloc(sizeof(double) * (size_t)V);
  double* lq = malloc(sizeof(double) * (size_t)V);
  if (!lp || !lq) {
    free(lp);
    free(lq);
    return ORC_ERR_MEM;
  }
  orc_row_target st;
  row_target(V, dtype, zp, zq, alpha, beta, T, lp, lq, logpi, &st);
  if (lse_p) *lse_p = st.lse_p;
  if (lse_q) *lse_q = st.lse_q;
  if (log_zcd) *log_zcd = st.log_zcd;
  if (cd_lse) *cd_lse = st.cd_lse;
  if (argmax) *argmax = st.argmax;
  if (gap_argmax) *gap_argmax = st.gap_argmax;
  free(lp);
  free(lq);
  return ORC_OK;
}

/*
 * The sibling-rejection chain of one row, run to the end as if every child were rejected:
 * ratios[j] = r_{j}(t_j) / q(t_j) for j = 0..m-1 (r_0 = pi_CD,T), and r_m in r_out[V].
 */
int dcd_oracle_row_chain(int64_t V, int dtype, const void* zp, const void* zq, double alpha, double beta,
                         double T, const float* q, int m, const int32_t* child_tokens, int distinct, double* ratios,
                         double* r_out) {
  if (V <= 0 || !zp || !zq || !q || m < 0 || !r_out || T <= 0.0) return ORC_ERR_ARG;
  double* lp = malloc(sizeof(double) * (size_t)V);
  double* lq = malloc(sizeof(double) * (size_t)V);
  double* tmp = malloc(sizeof(double) * (size_t)V);
  double* qd = distinct ? malloc(sizeof(double) * (size_t)V) : NULL;
  if (!lp || !lq || !tmp || (distinct && !qd)) {
    free(lp);
    free(lq);
    free(tmp);
    free(qd);
    return ORC_ERR_MEM;
  }
  orc_row_target st;
  row_target(V, dtype, zp, zq, alpha, beta, T, lp, lq, r_out, &st);
  for (int64_t x = 0; x < V; ++x) r_out[x] = exp(r_out[x]);
  if (distinct)
    for (int64_t x = 0; x < V; ++x) qd[x] = (double)q[x];
  for (int j = 0; j < m; ++j) {
    const int32_t t = child_tokens[j];
    if (distinct) {
      ratios[j] = accept_ratio(r_out[t], qd[t]);
      residual_step_d(V, r_out, qd, tmp);
      remove_token(V, qd, t);
    } else {
      ratios[j] = accept_ratio(r_out[t], (double)q[t]);
      residual_step(V, r_out, q, tmp);
    }
  }
  free(lp);
  free(lq);
  free(tmp);
  free(qd);
  return ORC_OK;
}

/* ---------------------------------------------------------------- full verification */

typedef struct {
  double cd_lse;       /* raw-logit normaliser at T_eff (library output cd_lse) */
  double log_zcd;      /* the paper's log Z_CD at T_eff */
  double gap_argmax;   /* top-2 score gap */
  double gap_mask;     /* distance to the plausibility threshold */
  double gap_accept;   /* min |u - ratio| / max(1, ratio) over the acceptance tests taken */
  double gap_race;     /* top-2 race-key gap (+inf when no race was run) */
  int32_t argmax;      /* argmax of the CD score on P_beta */
  int32_t acc_child;   /* accepted child node id, -1 if none */
  int32_t term_token;  /* terminal token (argmax or race winner) when acc_child < 0, else -1 */
  int32_t n_tests;     /* acceptance tests taken */
} dcd_oracle_row;

/*
 * Verifies B sequences of N tree nodes each.  Row g = b*N + n of z_p / z_q (row stride ld
 * elements; ld = 0 repeats one row) holds the logits after node n.  q (row stride ldq) is read
 * only for non-leaf rows of sequences with temperature > 0.  beta and temperature may be NULL
 * (all zero).  Outputs: accept_len[B], accept_path[B*N] (node ids, padded with -1), bonus[B],
 * cd_logprob[B*N] (log pi_CD,T_eff(token_n) under the parent's row, root 0), rows[B*N], and
 * residual[B*V] (optional: the distribution each sequence's bonus was drawn from; one-hot at
 * the argmax for greedy sequences).  seq_ids (may be NULL = 0..B-1) gives each sequence's index
 * in the batch it was drawn from; Philox counters use it, so a subset of a batch draws the same
 * uniforms as the whole batch.
 * Returns 0, or a negative code for invalid arguments / a malformed tree.
 */
int dcd_oracle_verify(int32_t B, int32_t N, int64_t V, int dtype, int64_t ld, const void* zp, const void* zq,
                      const int32_t* tokens, const int32_t* parents, const float* alpha, const float* beta,
                      const float* temperature, const float* q, int64_t ldq, uint64_t seed, uint64_t offset,
                      const int32_t* seq_ids, int distinct, int nthreads, int32_t* accept_len, int32_t* accept_path,
                      int32_t* bonus, double* cd_logprob, dcd_oracle_row* rows, double* residual) {
  if (B < 0 || N < 1 || V < 1 || (dtype < 0 || dtype > 2) || ld < 0 || !zp || !zq || !tokens || !parents ||
      !alpha || !accept_len || !accept_path || !bonus || !cd_logprob || !rows)
    return ORC_ERR_ARG;
  for (int32_t b = 0; b < B; ++b) {
    if (parents[(int64_t)b * N] != -1) return ORC_ERR_TREE;
    for (int32_t n = 1; n < N; ++n) {
      const int32_t p = parents[(int64_t)b * N + n];
      const int32_t t = tokens[(int64_t)b * N + n];
      if (p < 0 || p >= n || t < 0 || t >= V) return ORC_ERR_TREE;
    }
    if (temperature && (temperature[b] > 0.0f && !q)) return ORC_ERR_ARG;
    if (temperature && !(temperature[b] >= 0.0f)) return ORC_ERR_ARG;
    if (!(alpha[b] >= 0.0f)) return ORC_ERR_ARG;
    if (beta && !(beta[b] >= 0.0f && beta[b] <= 1.0f)) return ORC_ERR_ARG;
  }
  const size_t es = dtype_size(dtype);
  const int64_t R = (int64_t)B * N;
  int err = ORC_OK;
  if (nthreads < 1) nthreads = 1;

#pragma omp parallel num_threads(nthreads)
  {
    double* lp = malloc(sizeof(double) * (size_t)V);
    double* lq = malloc(sizeof(double) * (size_t)V);
    double* r = malloc(sizeof(double) * (size_t)V);
    double* tmp = malloc(sizeof(double) * (size_t)V);
    double* qd = malloc(sizeof(double) * (size_t)V);
    int32_t* kids = malloc(sizeof(int32_t) * (size_t)N);
    const int have_mem = lp && lq && r && tmp && qd && kids;
    if (!have_mem) {
#pragma omp atomic write
      err = ORC_ERR_MEM;
    }
    /* every thread reaches the work-sharing loop; one without scratch takes no work */
    {
#pragma omp for schedule(dynamic, 1)
      for (int64_t g = 0; g < R; ++g) {
        if (!have_mem) continue;
        const int32_t b = (int32_t)(g / N), n = (int32_t)(g % N);
        const double a = alpha[b];
        const double be = beta ? beta[b] : 0.0;
        const double T = temperature ? temperature[b] : 0.0;
        const char* zpr = (const char*)zp + (size_t)(ld * g) * es;
        const char* zqr = (const char*)zq + (size_t)(ld * g) * es;
        orc_row_target st;
        row_target(V, dtype, zpr, zqr, a, be, T, lp, lq, r, &st);
        dcd_oracle_row* out = &rows[g];
        out->cd_lse = st.cd_lse;
        out->log_zcd = st.log_zcd;
        out->gap_argmax = st.gap_argmax;
        out->gap_mask = st.gap_mask;
        out->gap_accept = INFINITY;
        out->gap_race = INFINITY;
        out->argmax = st.argmax;
        out->acc_child = -1;
        out->term_token = -1;
        out->n_tests = 0;
        /* children of node n, ascending node id */
        int m = 0;
        for (int32_t c = n + 1; c < N; ++c)
          if (parents[(int64_t)b * N + c] == n) kids[m++] = c;
        /* log-probabilities of the children's tokens under this row */
        for (int k = 0; k < m; ++k) {
          const int32_t c = kids[k];
          cd_logprob[(int64_t)b * N + c] = r[tokens[(int64_t)b * N + c]];
        }
        if (n == 0) cd_logprob[(int64_t)b * N] = 0.0;
        if (!(T > 0.0)) {
          /* greedy rule: first child (ascending id) whose token is the argmax */
          for (int k = 0; k < m && out->acc_child < 0; ++k)
            if (tokens[(int64_t)b * N + kids[k]] == st.argmax) out->acc_child = kids[k];
          if (out->acc_child < 0) out->term_token = st.argmax;
          continue;
        }
        /* sampled rule: r_0 = pi_CD,T; siblings drawn without replacement each see q without
           the tokens of the siblings rejected before them, renormalised */
        for (int64_t x = 0; x < V; ++x) r[x] = exp(r[x]);
        const float* qr = q + (size_t)(ldq * g);
        if (distinct)
          for (int64_t x = 0; x < V; ++x) qd[x] = (double)qr[x];
        for (int k = 0; k < m; ++k) {
          const int32_t c = kids[k];
          const int32_t t = tokens[(int64_t)b * N + c];
          const double ratio = distinct ? accept_ratio(r[t], qd[t]) : accept_ratio(r[t], (double)qr[t]);
          const int64_t sb = seq_ids ? seq_ids[b] : b;
          const double u = dcd_oracle_accept_uniform(seed, offset, (uint32_t)(sb * N + c));
          ++out->n_tests;
          if (isfinite(ratio)) {
            const double d = fabs(u - ratio) / (ratio > 1.0 ? ratio : 1.0);
            if (d < out->gap_accept) out->gap_accept = d;
          }
          if (u <= ratio) {
            out->acc_child = c;
            break;
          }
          if (distinct) {
            residual_step_d(V, r, qd, tmp);
            remove_token(V, qd, t);
          } else {
            residual_step(V, r, qr, tmp);
          }
        }
        if (out->acc_child < 0) {
          const int64_t sb = seq_ids ? seq_ids[b] : b;
          out->term_token = race(V, r, seed, offset, (uint32_t)(sb * N + n), &out->gap_race);
        }
      }
    }
    free(lp);
    free(lq);
    free(r);
    free(tmp);
    free(qd);
    free(kids);
  }
  if (err) return err;

  /* tree walk */
  for (int32_t b = 0; b < B; ++b) {
    int32_t* path = accept_path + (int64_t)b * N;
    for (int32_t i = 0; i < N; ++i) path[i] = -1;
    int32_t cur = 0, len = 0;
    path[0] = 0;
    while (rows[(int64_t)b * N + cur].acc_child >= 0) {
      cur = rows[(int64_t)b * N + cur].acc_child;
      path[++len] = cur;
    }
    accept_len[b] = len;
    bonus[b] = rows[(int64_t)b * N + cur].term_token;
    if (residual) {
      double* res = residual + (size_t)b * (size_t)V;
      const double T = temperature ? temperature[b] : 0.0;
      if (!(T > 0.0)) {
        for (int64_t x = 0; x < V; ++x) res[x] = 0.0;
        res[bonus[b]] = 1.0;
        continue;
      }
      /* recompute the terminal residual of the last node's row: every child was rejected */
      double* lp = malloc(sizeof(double) * (size_t)V);
      double* lq = malloc(sizeof(double) * (size_t)V);
      double* tmp = malloc(sizeof(double) * (size_t)V);
      double* qd = malloc(sizeof(double) * (size_t)V);
      if (!lp || !lq || !tmp || !qd) {
        free(lp);
        free(lq);
        free(tmp);
        free(qd);
        return ORC_ERR_MEM;
      }
      const int64_t g = (int64_t)b * N + cur;
      orc_row_target st;
      row_target(V, dtype, (const char*)zp + (size_t)(ld * g) * es, (const char*)zq + (size_t)(ld * g) * es,
                 alpha[b], beta ? beta[b] : 0.0, T, lp, lq, res, &st);
      for (int64_t x = 0; x < V; ++x) res[x] = exp(res[x]);
      const float* qr = q + (size_t)(ldq * g);
      for (int64_t x = 0; x < V; ++x) qd[x] = (double)qr[x];
      for (int32_t c = cur + 1; c < N; ++c) {
        if (parents[(int64_t)b * N + c] != cur) continue;
        if (distinct) {
          residual_step_d(V, res, qd, tmp);
          remove_token(V, qd, tokens[(int64_t)b * N + c]);
        } else {
          residual_step(V, res, qr, tmp);
        }
      }
      free(lp);
      free(lq);
      free(tmp);
      free(qd);
    }
  }
  return ORC_OK;
}

int dcd_oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* ---------------------------------------------------------------- per-row diagnostics */

/*
 * Diagnostics of one row (the quantities of the paper's signal--proposal-error diagnostic,
 * Sec. 3.1, of its alignment-gap estimator, App. C, and of the KL decomposition of App. B), in
 * fp64 from the exact inputs:
 *   lse_p, lse_q : log sum_x exp(z_p(x)), log sum_x exp(z_q(x)) (full vocabulary);
 *   signal       : |log pi_p(x*) - log pi_q(x*)| at the given token x* (the CD argmax);
 *   e_q          : E_{pi_q}[log pi_p - log pi_q];
 *   e_e, kl_e_p  : with the drafter's distribution pi_e = q (q may be NULL): E_{pi_e}[log pi_p -
 *                  log pi_q] and D_KL(pi_e || pi_p), with 0 log 0 = 0;
 *   kl_p_q       : D_KL(pi_p || pi_q) = E_{pi_p}[log pi_p - log pi_q];
 *   kl_p_cd      : D_KL(pi_p || pi_CD) for the untruncated, untempered target of Eq. 1,
 *                  pi_CD proportional to pi_p^(1 + alpha) pi_q^(-alpha) over the whole vocabulary,
 *                  summed term by term from that definition (NaN when alpha < 0: not requested).
 * out[8] = {lse_p, lse_q, signal, e_q, e_e, kl_e_p, kl_p_q, kl_p_cd} (e_e, kl_e_p NaN without q).
 */
int dcd_oracle_row_diagnostics(int64_t V, int dtype, const void* zp, const void* zq, const float* q, int32_t xstar,
                               double alpha, double* out) {
  if (V <= 0 || !zp || !zq || !out || xstar < 0 || xstar >= V) return ORC_ERR_ARG;
  double mp = -INFINITY, mq = -INFINITY;
  for (int64_t x = 0; x < V; ++x) {
    const double a = logit_at(zp, dtype, x), b = logit_at(zq, dtype, x);
    if (a > mp) mp = a;
    if (b > mq) mq = b;
  }
  double sp = 0.0, sq = 0.0;
  for (int64_t x = 0; x < V; ++x) {
    sp += exp(logit_at(zp, dtype, x) - mp);
    sq += exp(logit_at(zq, dtype, x) - mq);
  }
  const double lse_p = mp + log(sp), lse_q = mq + log(sq);
  double e_q = 0.0, e_e = 0.0, kl = 0.0, kl_pq = 0.0;
  for (int64_t x = 0; x < V; ++x) {
    const double lp = logit_at(zp, dtype, x) - lse_p, lq = logit_at(zq, dtype, x) - lse_q;
    e_q += exp(lq) * (lp - lq);
    kl_pq += exp(lp) * (lp - lq);
    if (q) {
      const double e = (double)q[x];
      e_e += e * (lp - lq);
      if (e > 0.0) kl += e * (log(e) - lp);
    }
  }
  double kl_cd = NAN;
  if (alpha >= 0.0) {
    /* log pi_CD(x) = (1 + alpha) lp(x) - alpha lq(x) - log Z_CD (Eq. 1 with beta = 0, T = 1) */
    double ms = -INFINITY;
    for (int64_t x = 0; x < V; ++x) {
      const double lp = logit_at(zp, dtype, x) - lse_p, lq = logit_at(zq, dtype, x) - lse_q;
      const double sc = (1.0 + alpha) * lp - alpha * lq;
      if (sc > ms) ms = sc;
    }
    double ss = 0.0;
    for (int64_t x = 0; x < V; ++x) {
      const double lp = logit_at(zp, dtype, x) - lse_p, lq = logit_at(zq, dtype, x) - lse_q;
      ss += exp((1.0 + alpha) * lp - alpha * lq - ms);
    }
    const double log_z = ms + log(ss);
    kl_cd = 0.0;
    for (int64_t x = 0; x < V; ++x) {
      const double lp = logit_at(zp, dtype, x) - lse_p, lq = logit_at(zq, dtype, x) - lse_q;
      const double lcd = (1.0 + alpha) * lp - alpha * lq - log_z;
      kl_cd += exp(lp) * (lp - lcd);
    }
  }
  out[0] = lse_p;
  out[1] = lse_q;
  out[2] = fabs((logit_at(zp, dtype, xstar) - lse_p) - (logit_at(zq, dtype, xstar) - lse_q));
  out[3] = e_q;
  out[4] = q ? e_e : NAN;
  out[5] = q ? kl : NAN;
  out[6] = kl_pq;
  out[7] = kl_cd;
  return ORC_OK;
}
