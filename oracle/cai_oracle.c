/*
 * CAI-dLLM oracle: TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, deliberately unoptimised CPU statement of what one denoising
 * step of the CAI-dLLM decoding head computes (arXiv 2608.22646, Section 4):
 *
 *   - the decoding head of Box 1 ("Token Confidence"): logits z = W h for each
 *     masked position, the full-vocabulary softmax, the confidence
 *     c = max_v p(v) and the greedy token argmax_v p(v);
 *   - the confidence-aware controller of Boxes 2-7 and Algorithm 1: first-step
 *     confidence s_i (Box 2), the cosine threshold schedule (Box 3) with the
 *     block-specific end threshold (Box 4), the confidence-gated token budget
 *     (Box 5, Eq. token_budget), the position-aware threshold and commit rule
 *     (Box 6, Eqs. position_threshold and position_commit), and the grinding
 *     phase detector with its force-commit threshold (Box 7,
 *     Eq. grinding-detector), gated as in Section 4.6.
 *
 * Everything is IEEE double.  bf16 inputs are decoded by this file's own bit
 * shift.  Dot products accumulate in ascending k order; the softmax is the
 * textbook two-pass one (max, then sum of exponentials).  There is no
 * blocking, fusion or reordering.  Rows may run on separate threads, but
 * each row is computed by one thread from start to end.
 *
 * Nothing under the product package includes, links or calls this file, and
 * this file includes nothing from it.  Only the tests, the smoke check, the
 * benchmark's CPU-baseline leg and reference arm, and the generator
 * calibration script beside this file load it.
 *
 * Readings of points the paper leaves open (each selectable by a flag):
 *   - eta_bar (Box 7): count mode reads "eta < 1.5" as a count of newly
 *     committed tokens, as Algorithm 1 counts them.  Fraction mode reads it as
 *     eta / L < eta_bar with L the generation length.
 *   - theta_e^(b) for b > 4 (Box 4): floored at theta_e_min (0.40, the b = 4
 *     value).  CAI_O_QUARTER_BLOCKS maps block b to the quarter of the output
 *     that it falls in.
 *   - position and budget tiers (Boxes 5, 6): absolute as printed (16/32/48).
 *     CAI_O_QUARTER_POS scales them to P/4, P/2, 3P/4.
 *   - warm-up (Box 3, t < wT): tested exactly as 100 t < warmup_pct T.
 *   - gating OFF (Section 4.6): no budgets, no grinding exit and no
 *     force commit; the position factors stay.
 *   - tokens still masked when a block exits stay masked unless
 *     CAI_O_FLUSH_ON_EXIT is set, which commits them to their current argmax
 *     without counting them in eta.
 *   - ties: argmax takes the lowest vocabulary index; c >= theta_i is
 *     inclusive; c > theta_fb is strict.
 *   - order inside a step (Algorithm 1): commit loop, eta, the low-yield
 *     counter, the grinding check, then the "nothing masked" check; a block
 *     that reaches t = T - 1 without either exit is "T exhausted".
 *   - the batch runs blocks and steps in lockstep; each sequence keeps its
 *     own low-yield counter and exit state.
 *
 * Ablation variants (Section 5.3, Table "HumanEval ablation"):
 *   - CAI_O_NO_BLOCK_SCHEDULE: Box 3 alone ("APD"): every block ends at
 *     theta_e1 = 0.70 instead of Box 4's theta_e^(b).
 *   - CAI_O_FIXED_THRESHOLD: the fixed-threshold rule of Fast-dLLM that the
 *     paper compares with: theta^(b)(t) = theta_s for every step and block.
 *
 * Diagnostics (Section 2.1, CAI_O_DIAGNOSTICS):
 *   - the stability step t_i^*: a token is stable once its top prediction has
 *     been the same at three consecutive steps; t_i^* is the local step of the
 *     third of them (read here as the step at which stability is first
 *     observed).  Only steps that decode the token count: a token committed
 *     before that has no t_i^* (-1).
 *   - the relative L2 drift D^(t) = mean over the block's positions of
 *     ||h^(t) - h^(t-1)|| / ||h^(t-1)|| (Eq. relative_drift), per sequence,
 *     from the hidden states of consecutive steps of one block (cai_o_drift).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define CAI_O_GATING 1u
#define CAI_O_POS_FACTOR 2u
#define CAI_O_FLUSH_ON_EXIT 4u
#define CAI_O_QUARTER_POS 8u
#define CAI_O_QUARTER_BLOCKS 16u
#define CAI_O_NO_BLOCK_SCHEDULE 32u
#define CAI_O_FIXED_THRESHOLD 64u
#define CAI_O_DIAGNOSTICS 128u

#define CAI_O_MASK (-1)

enum { CAI_O_RUNNING = 0, CAI_O_EXIT_DONE = 1, CAI_O_EXIT_GRIND = 2, CAI_O_EXIT_TMAX = 3 };

typedef struct {
  int32_t B, P, T, n_blocks;
  double theta_s;      /* Box 3: start threshold, 0.90 */
  double theta_e1;     /* Box 4: end threshold of block 1, 0.70 */
  double theta_e_step; /* Box 4: decrease per block, 0.10 */
  double theta_e_min;  /* floor for b > 4, 0.40 */
  int32_t warmup_pct;  /* Box 3: w = 0.15 as a percentage */
  int32_t K;           /* Box 7: patience window, 4 */
  double theta_fb;     /* Box 7: force-commit threshold, 0.40 */
  double clip_lo;      /* Box 6: 0.20 */
  double clip_hi;      /* Box 6: 0.98 */
  double eta_bar;      /* Box 7: 1.5 (count mode) or 0.015 (fraction mode) */
  int32_t eta_mode;    /* 0 = count, 1 = fraction of generation length */
  uint32_t flags;
} cai_o_cfg;

/* ---------------------------------------------------------------- bf16 -- */

/* A bf16 value is the upper half of an IEEE binary32; widening is exact. */
double cai_o_bf16_to_double(uint16_t bits) {
  uint32_t u = ((uint32_t)bits) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* ------------------------------------------------------ decoding head -- */

/* Box 1 for one row h of length H against every row of W [V, H]:
 *   z_v = sum_k W[v,k] x[k], with x = h, or, when the model's final RMSNorm is
 *   part of the head (g != NULL), x[k] = g[k] h[k] / r, r = sqrt(sum_k h[k]^2 / H + eps)
 *   m   = max_v z_v, idx = lowest v with z_v = m
 *   S   = sum_v exp(z_v - m),  c = max_v p_v = exp(m - LSE) = 1 / S
 * gap = m - (largest z_v over v != idx), +inf when V = 1. */
static void head_one_row(const uint16_t* W, int32_t V, int32_t H, const uint16_t* h,
                         const uint16_t* g, double eps, double* x, double* z, double* conf,
                         int32_t* argmax, double* zmax, double* lse, double* gap) {
  for (int32_t k = 0; k < H; ++k) x[k] = cai_o_bf16_to_double(h[k]);
  if (g) {
    double ss = 0.0;
    for (int32_t k = 0; k < H; ++k) ss += x[k] * x[k];
    const double r = sqrt(ss / (double)H + eps);
    for (int32_t k = 0; k < H; ++k) x[k] = cai_o_bf16_to_double(g[k]) * x[k] / r;
  }
  for (int32_t v = 0; v < V; ++v) {
    const uint16_t* w = W + (size_t)v * (size_t)H;
    double acc = 0.0;
    for (int32_t k = 0; k < H; ++k) acc += cai_o_bf16_to_double(w[k]) * x[k];
    z[v] = acc;
  }
  double m = z[0];
  int32_t idx = 0;
  for (int32_t v = 1; v < V; ++v) {
    if (z[v] > m) {
      m = z[v];
      idx = v;
    }
  }
  double second = -INFINITY;
  for (int32_t v = 0; v < V; ++v) {
    if (v != idx && z[v] > second) second = z[v];
  }
  double S = 0.0;
  for (int32_t v = 0; v < V; ++v) S += exp(z[v] - m);
  *conf = 1.0 / S;
  *argmax = idx;
  *zmax = m;
  *lse = m + log(S);
  *gap = m - second;
}

typedef struct {
  const uint16_t* W;
  int32_t V, H;
  const uint16_t* rows;
  const uint16_t* g;
  double eps;
  int32_t M, first, stride;
  double *conf, *zmax, *lse, *gap;
  int32_t* argmax;
  int32_t failed;
} head_job;

static void* head_worker(void* arg) {
  head_job* j = (head_job*)arg;
  double* z = (double*)malloc(sizeof(double) * (size_t)j->V);
  double* x = (double*)malloc(sizeof(double) * (size_t)j->H);
  if (!z || !x) {
    free(z);
    free(x);
    j->failed = 1;
    return NULL;
  }
  for (int32_t i = j->first; i < j->M; i += j->stride) {
    head_one_row(j->W, j->V, j->H, j->rows + (size_t)i * (size_t)j->H, j->g, j->eps, x, z,
                 &j->conf[i], &j->argmax[i], &j->zmax[i], &j->lse[i], &j->gap[i]);
  }
  free(z);
  free(x);
  return NULL;
}

/* Decoding head over M rows [M, H], with the model's final RMSNorm (weight g
 * [H], epsilon eps) applied to each row first when g is not NULL.  Rows are
 * spread over n_threads threads; each row is computed start to end by one
 * thread.  Returns 0 on success. */
int32_t cai_o_head_rows_norm(const uint16_t* W, int32_t V, int32_t H, const uint16_t* rows,
                             int32_t M, const uint16_t* g, double eps, int32_t n_threads,
                             double* conf, int32_t* argmax, double* zmax, double* lse, double* gap) {
  if (V <= 0 || H <= 0 || M < 0) return -1;
  if (M == 0) return 0;
  if (n_threads < 1) n_threads = 1;
  if (n_threads > M) n_threads = M;
  head_job* jobs = (head_job*)calloc((size_t)n_threads, sizeof(head_job));
  pthread_t* th = (pthread_t*)calloc((size_t)n_threads, sizeof(pthread_t));
  if (!jobs || !th) {
    free(jobs);
    free(th);
    return -2;
  }
  int32_t rc = 0;
  for (int32_t t = 0; t < n_threads; ++t) {
    head_job j = {W, V, H, rows, g, eps, M, t, n_threads, conf, zmax, lse, gap, argmax, 0};
    jobs[t] = j;
  }
  int32_t started = 0;
  for (int32_t t = 1; t < n_threads; ++t) {
    if (pthread_create(&th[t], NULL, head_worker, &jobs[t]) != 0) break;
    started = t;
  }
  head_worker(&jobs[0]);
  for (int32_t t = 1; t <= started; ++t) pthread_join(th[t], NULL);
  /* Any job whose thread could not start runs here. */
  for (int32_t t = started + 1; t < n_threads; ++t) head_worker(&jobs[t]);
  for (int32_t t = 0; t < n_threads; ++t)
    if (jobs[t].failed) rc = -2;
  free(jobs);
  free(th);
  return rc;
}

/* Full probability vector of one row (for the sum-to-one and brute-force
 * pins): p_v = exp(z_v - m) / S. */
/* Box 1 without the final RMSNorm. */
int32_t cai_o_head_rows(const uint16_t* W, int32_t V, int32_t H, const uint16_t* rows, int32_t M,
                        int32_t n_threads, double* conf, int32_t* argmax, double* zmax, double* lse,
                        double* gap) {
  return cai_o_head_rows_norm(W, V, H, rows, M, NULL, 0.0, n_threads, conf, argmax, zmax, lse, gap);
}

int32_t cai_o_softmax_row(const uint16_t* W, int32_t V, int32_t H, const uint16_t* h, double* z_out,
                          double* p_out) {
  double conf, zmax, lse, gap;
  int32_t idx;
  double* x = (double*)malloc(sizeof(double) * (size_t)H);
  if (!x) return -1;
  head_one_row(W, V, H, h, NULL, 0.0, x, z_out, &conf, &idx, &zmax, &lse, &gap);
  free(x);
  double S = 0.0;
  for (int32_t v = 0; v < V; ++v) S += exp(z_out[v] - zmax);
  for (int32_t v = 0; v < V; ++v) p_out[v] = exp(z_out[v] - zmax) / S;
  return idx;
}

/* ------------------------------------------------------- thresholds -- */

/* Box 4: theta_e^(b) = 0.70 - 0.10 (b - 1) for the 1-based block index b,
 * floored at theta_e_min.  Quarter mode: b -> 1 + floor(4 (b - 1) / n_blocks). */
double cai_o_theta_e(const cai_o_cfg* c, int32_t b) {
  int32_t be = b;
  if (c->flags & CAI_O_QUARTER_BLOCKS) be = 1 + (4 * (b - 1)) / c->n_blocks;
  if (c->flags & CAI_O_NO_BLOCK_SCHEDULE) be = 1;
  double th = c->theta_e1 - c->theta_e_step * (double)(be - 1);
  if (th < c->theta_e_min) th = c->theta_e_min;
  return th;
}

/* Boxes 3 and 4: theta^(b)(t) = theta_s while t < wT, else
 * theta_e^(b) + (theta_s - theta_e^(b))/2 (1 + cos(pi (t - wT) / (T - wT))). */
double cai_o_theta_block(const cai_o_cfg* c, int32_t b, int32_t t) {
  if (c->flags & CAI_O_FIXED_THRESHOLD) return c->theta_s;
  if (100 * t < c->warmup_pct * c->T) return c->theta_s;
  const double pi = 3.14159265358979323846;
  double wT = (double)c->warmup_pct * (double)c->T / 100.0;
  double u = ((double)t - wT) / ((double)c->T - wT);
  double te = cai_o_theta_e(c, b);
  double alpha = (c->theta_s - te) / 2.0;
  return te + alpha * (1.0 + cos(pi * u));
}

/* Box 6: r_pos(i) = 0.80 / 0.90 / 1.05 / 1.10 for p < 16 / < 32 / < 48 / >= 48. */
double cai_o_pos_factor(const cai_o_cfg* c, int32_t p) {
  if (!(c->flags & CAI_O_POS_FACTOR)) return 1.0;
  int32_t q1 = 16, q2 = 32, q3 = 48;
  if (c->flags & CAI_O_QUARTER_POS) {
    q1 = c->P / 4;
    q2 = c->P / 2;
    q3 = (3 * c->P) / 4;
  }
  if (p < q1) return 0.80;
  if (p < q2) return 0.90;
  if (p < q3) return 1.05;
  return 1.10;
}

/* Box 6, Eq. position_threshold: theta_i(t) = clip(theta_b(t) r_pos(i), 0.20, 0.98). */
double cai_o_theta_token(const cai_o_cfg* c, int32_t b, int32_t t, int32_t p) {
  double th = cai_o_theta_block(c, b, t) * cai_o_pos_factor(c, p);
  if (th < c->clip_lo) th = c->clip_lo;
  if (th > c->clip_hi) th = c->clip_hi;
  return th;
}

/* Box 5, Eq. token_budget, cases in order:
 *   8 if s > 0.50 and p < 32;  64 if s < 0.25 or p >= 48;  32 otherwise. */
int32_t cai_o_budget(const cai_o_cfg* c, double s, int32_t p) {
  int32_t half = 32, late = 48;
  if (c->flags & CAI_O_QUARTER_POS) {
    half = c->P / 2;
    late = (3 * c->P) / 4;
  }
  if (s > 0.50 && p < half) return 8;
  if (s < 0.25 || p >= late) return 64;
  return 32;
}

/* Box 7: is a step that committed eta tokens a low-yield step? */
int32_t cai_o_low_yield(const cai_o_cfg* c, int32_t eta) {
  if (c->eta_mode == 1) {
    double L = (double)c->n_blocks * (double)c->P;
    return ((double)eta / L) < c->eta_bar;
  }
  return (double)eta < c->eta_bar;
}

/* ------------------------------------------------------- controller -- */

typedef struct {
  int32_t* tok;         /* [B, L] committed token, -1 = MASK; L = n_blocks P */
  double* conf;         /* [B, L] confidence at the last step that saw the token masked */
  double* s0;           /* [B, L] first-step confidence s_i (Box 2) */
  int32_t* budget;      /* [B, L] B_i (Box 5); 0 before the block starts */
  int32_t* cstep;       /* [B, L] local step of the commit, -1 = not committed */
  int32_t* cand;        /* [B, L] argmax at the last step that saw the token masked */
  int32_t* ell;         /* [B] low-yield counter (Algorithm 1) */
  int32_t* eta;         /* [B] tokens committed by the commit rule at the last step */
  int32_t* exit_reason; /* [B, n_blocks] 0 running, 1 done, 2 grinding, 3 T exhausted */
  int32_t* exit_step;   /* [B, n_blocks] local step at which the block exited, -1 */
  int32_t* unresolved;  /* [B, n_blocks] tokens left masked at exit */
  int32_t* run;         /* [B, L] consecutive decoded steps with the same top prediction */
  int32_t* stable;      /* [B, L] stability step t_i^*, -1 = not (yet) stable */
} cai_o_state;

/* One denoising step of Algorithm 1 for every running sequence of the batch,
 * at local step t of block blk (0-based; the paper's b = blk + 1).
 * conf_in/idx_in hold c_i^(t) and argmax_v p for every position (b, p) of the
 * current block, [B, P]; only entries of still-masked tokens of running
 * sequences are read. */
void cai_o_controller_step(const cai_o_cfg* c, cai_o_state* st, int32_t blk, int32_t t,
                           const double* conf_in, const int32_t* idx_in) {
  const int32_t B = c->B, P = c->P, L = c->n_blocks * c->P;
  const int32_t gating = (c->flags & CAI_O_GATING) != 0;
  for (int32_t b = 0; b < B; ++b) {
    const int32_t eb = b * c->n_blocks + blk;
    if (st->exit_reason[eb] != CAI_O_RUNNING) continue;
    if (t == 0) st->ell[b] = 0; /* Algorithm 1: ell <- 0 before the block's first step */
    int32_t eta = 0;
    /* commit loop: foreach masked token i */
    for (int32_t p = 0; p < P; ++p) {
      const int32_t g = b * L + blk * P + p;
      if (st->tok[g] != CAI_O_MASK) continue;
      const double ci = conf_in[b * P + p];
      const int32_t xi = idx_in[b * P + p];
      if (t == 0) {
        st->s0[g] = ci;
        st->budget[g] = cai_o_budget(c, ci, p);
      }
      if (c->flags & CAI_O_DIAGNOSTICS) {
        st->run[g] = (t > 0 && st->cand[g] == xi) ? st->run[g] + 1 : 1;
        if (st->run[g] >= 3 && st->stable[g] < 0) st->stable[g] = t;
      }
      st->conf[g] = ci;
      st->cand[g] = xi;
      const double th = cai_o_theta_token(c, blk + 1, t, p);
      const int32_t by_conf = ci >= th;
      const int32_t by_budget = gating && t >= st->budget[g];
      if (by_conf || by_budget) {
        st->tok[g] = xi;
        st->cstep[g] = t;
        eta += 1;
      }
    }
    st->eta[b] = eta;
    /* low-yield counter */
    if (cai_o_low_yield(c, eta))
      st->ell[b] += 1;
    else
      st->ell[b] = 0;
    int32_t reason = CAI_O_RUNNING;
    if (gating && st->ell[b] >= c->K) {
      /* grinding phase: force-commit the masked tokens with c > theta_fb */
      for (int32_t p = 0; p < P; ++p) {
        const int32_t g = b * L + blk * P + p;
        if (st->tok[g] == CAI_O_MASK && st->conf[g] > c->theta_fb) {
          st->tok[g] = st->cand[g];
          st->cstep[g] = t;
        }
      }
      reason = CAI_O_EXIT_GRIND;
    } else {
      int32_t left = 0;
      for (int32_t p = 0; p < P; ++p)
        if (st->tok[b * L + blk * P + p] == CAI_O_MASK) ++left;
      if (left == 0)
        reason = CAI_O_EXIT_DONE;
      else if (t == c->T - 1)
        reason = CAI_O_EXIT_TMAX;
    }
    if (reason != CAI_O_RUNNING) {
      int32_t left = 0;
      for (int32_t p = 0; p < P; ++p) {
        const int32_t g = b * L + blk * P + p;
        if (st->tok[g] != CAI_O_MASK) continue;
        if (c->flags & CAI_O_FLUSH_ON_EXIT) {
          st->tok[g] = st->cand[g];
          st->cstep[g] = t;
        } else {
          ++left;
        }
      }
      st->exit_reason[eb] = reason;
      st->exit_step[eb] = t;
      st->unresolved[eb] = left;
    }
  }
}

/* Eq. relative_drift for one sequence: the mean over the P positions of
 * ||h_cur[p] - h_prev[p]||_2 / ||h_prev[p]||_2 (bf16 rows [P, H], fp64). */
double cai_o_drift(const uint16_t* h_prev, const uint16_t* h_cur, int32_t P, int32_t H) {
  double sum = 0.0;
  for (int32_t p = 0; p < P; ++p) {
    double num = 0.0, den = 0.0;
    for (int32_t k = 0; k < H; ++k) {
      const double a = cai_o_bf16_to_double(h_prev[(size_t)p * H + k]);
      const double d = cai_o_bf16_to_double(h_cur[(size_t)p * H + k]) - a;
      num += d * d;
      den += a * a;
    }
    sum += sqrt(num) / sqrt(den);
  }
  return sum / (double)P;
}
