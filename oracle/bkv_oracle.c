/*
 * BeaconKV compression step: plain fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call this file:
 * only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline / reference
 * leg load the shared library built from it.  It shares no code, header,
 * table or constant with the CUDA library (paper_2609_04971_gb300/csrc).
 *
 * Every function restates one step of the method as written in the paper
 * (BeaconKV, arXiv 2609.04971), in fp64, with plain loops in the order the
 * definitions are written.  Library primitives used as steps: libm sqrt, exp,
 * log, pow, cos, sin and qsort.
 *
 * Build flags matter: -ffp-contract=off (no fused multiply-add may change a
 * rounding), no -ffast-math.
 *
 * Conventions shared with the test harness (interfaces, not arithmetic):
 *   bf16 values are passed as raw uint16 bit patterns.
 *   One "instance" is one (layer, batch, KV head); its G query heads form the
 *   GQA group.  Group query sets are flattened head-major: row = h * n + i.
 *
 * Readings of points the paper leaves open:
 *   - beacons are kept per KV head and fed by all G query heads of its group;
 *     they are maintained as running-mean centroids seeded by FPS; in the
 *     Continual FPS mode they are instead each query head's fill-and-compress
 *     buffer (Eq. 9), compressed by the same fp64 FPS (Algorithm 1);
 *   - cosine with a zero vector is 0 (FPS) / the query is skipped (assignment);
 *   - argmin / argmax ties go to the lowest index;
 *   - RoPE uses the rotate-half pairing (i, i + d/2) with
 *     inv_freq_i = theta^(-2i/d); theta == 0 disables rotation;
 *   - scoring queries are rounded fp64 -> fp32 -> bf16 (round to nearest even);
 *   - the softmax runs over all L cached keys, with no mask; an optional causal
 *     mask inside the recent window takes positions: recent query w sits at
 *     recent_pos[w], beacons at the current step t, window key j (the last W
 *     rows) at t - (L - 1 - j), older keys before every window position;
 *   - top-k order is (score descending, index ascending).
 *
 * Parity pins for every function live in tests/test_oracle_*.py.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------ */
/* bf16 <-> binary64                                                   */
/* ------------------------------------------------------------------ */

/* A bf16 value is the top 16 bits of an IEEE binary32; widening is exact. */
double bkvo_bf16_to_f64(uint16_t h) {
  uint32_t u = ((uint32_t)h) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* binary32 -> bf16, round to nearest, ties to even (NaN kept quiet). */
uint16_t bkvo_f32_to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x007fffffu) != 0u)
    return (uint16_t)((u >> 16) | 0x0040u);
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7fffu + lsb;
  return (uint16_t)(u >> 16);
}

/* fp64 value -> fp32 (round to nearest even) -> bf16 (round to nearest even),
 * returned widened back to fp64.  This is the rounding of a scoring query. */
double bkvo_round_scoring(double x) {
  float f = (float)x;
  return bkvo_bf16_to_f64(bkvo_f32_to_bf16(f));
}

/* ------------------------------------------------------------------ */
/* Cosine similarity (Section 3.2; Appendix D.1)                       */
/* ------------------------------------------------------------------ */

static double dot_seq(const double* a, const double* b, int d) {
  double s = 0.0;
  for (int i = 0; i < d; ++i) s = s + a[i] * b[i];
  return s;
}

/* cos(a, b) = a.b / (|a| |b|), with |x| = sqrt(x.x); the sums run over i in
 * increasing order.  Returns 0 and sets *defined = 0 when a norm is zero. */
static double cosine(const double* a, const double* b, int d, int* defined) {
  double na = sqrt(dot_seq(a, a, d));
  double nb = sqrt(dot_seq(b, b, d));
  if (na == 0.0 || nb == 0.0) {
    if (defined) *defined = 0;
    return 0.0;
  }
  if (defined) *defined = 1;
  return dot_seq(a, b, d) / (na * nb);
}

double bkvo_cosine(const double* a, const double* b, int d) {
  return cosine(a, b, d, NULL);
}

static double* widen_rows(const uint16_t* q, int n, int d) {
  double* x = (double*)malloc(sizeof(double) * (size_t)n * (size_t)d);
  for (size_t i = 0; i < (size_t)n * (size_t)d; ++i) x[i] = bkvo_bf16_to_f64(q[i]);
  return x;
}

/* ------------------------------------------------------------------ */
/* Farthest Point Sampling (Appendix D.1, Algorithm 1)                 */
/* ------------------------------------------------------------------ */

/*
 * Selects m of the N pre-RoPE queries q (bf16, [N][d]).
 *   avg_i = (1/N) sum_j cos(q_i, q_j)        (j = i included)
 *   p     = argmin_i avg_i
 *   S_j   = cos(q_j, q_p)
 *   while fewer than m picked:
 *     r   = argmin over unpicked j of S_j;   pick r
 *     S_j = max(S_j, cos(q_j, q_r)) for the unpicked j
 * Ties go to the lowest index.  picks[k] is the k-th selected row.  gap[k] is
 * the distance from the minimum of step k to the runner-up value (+inf when
 * there is none) and alt[k] the runner-up's row (-1 when there is none): the
 * parity tests use them to recognise near-ties.
 *
 * Adoption (test harness only): where forced is not NULL and forced[k] >= 0,
 * step k takes row forced[k] instead of the argmin - the choice another
 * implementation, whose similarities carry rounding errors, may make at a
 * near-tie - and the farthest-point loop continues from it.  margin[k]
 * receives the value of the row taken minus the minimum (0 for the argmin),
 * and vals[k * N + j] the value step k minimises for row j (+inf for rows
 * picked before it).  A forced row that is out of range or already picked
 * makes the call return -1.  alt, margin and vals may be NULL.
 * Returns the number of picks (min(m, N)).
 */
int bkvo_fps_adopt(const uint16_t* q, int N, int d, int m, const int32_t* forced, int32_t* picks, double* gap,
                   int32_t* alt, double* margin, double* vals) {
  if (m > N) m = N;
  if (m <= 0) return 0;
  double* x = widen_rows(q, N, d);
  double* val = (double*)malloc(sizeof(double) * (size_t)N); /* the quantity minimised at the current step */
  char* sel = (char*)calloc((size_t)N, 1);
  int got = m;

  /* step 0 minimises the average cosine similarity of every query to the whole set */
  for (int i = 0; i < N; ++i) {
    double sum = 0.0;
    for (int j = 0; j < N; ++j) sum = sum + cosine(x + (size_t)i * d, x + (size_t)j * d, d, NULL);
    val[i] = sum / (double)N;
  }
  for (int k = 0; k < m; ++k) {
    int r = -1, r2 = -1;
    double b1 = INFINITY, b2 = INFINITY;
    for (int j = 0; j < N; ++j) {
      if (sel[j]) continue;
      if (val[j] < b1) {
        b2 = b1;
        r2 = r;
        b1 = val[j];
        r = j;
      } else if (val[j] < b2) {
        b2 = val[j];
        r2 = j;
      }
    }
    if (r < 0) { /* only reachable with non-finite inputs */
      got = k;
      break;
    }
    if (vals)
      for (int j = 0; j < N; ++j) vals[(size_t)k * N + j] = sel[j] ? INFINITY : val[j];
    int c = r;
    if (forced && forced[k] >= 0) {
      c = forced[k];
      if (c >= N || sel[c]) {
        got = -1;
        break;
      }
    }
    picks[k] = c;
    gap[k] = b2 - b1;
    if (alt) alt[k] = r2;
    if (margin) margin[k] = val[c] - b1;
    sel[c] = 1;
    /* S_j: the similarity to the first pick, then the running maximum over the picks */
    for (int j = 0; j < N; ++j) {
      if (sel[j]) continue;
      double cj = cosine(x + (size_t)j * d, x + (size_t)c * d, d, NULL);
      if (k == 0 || cj > val[j]) val[j] = cj;
    }
  }
  free(sel);
  free(val);
  free(x);
  return got;
}

int bkvo_fps(const uint16_t* q, int N, int d, int m, int32_t* picks, double* gap) {
  return bkvo_fps_adopt(q, N, d, m, NULL, picks, gap, NULL, NULL, NULL);
}

/* ------------------------------------------------------------------ */
/* Continual FPS (Section 4.2, Eq. 9; Algorithm 2 decode branch)       */
/* ------------------------------------------------------------------ */

/*
 * The fill-and-compress buffer of one query head (Eq. 9): every new query is
 * appended in order; when the buffer holds b_max queries it is replaced by
 * its FPS selection (Algorithm 1, fp64 similarities as in bkvo_fps) of b_min
 * queries, in pick order.
 *   buf     bf16 [b_max][d], rows [0, *size) in use; updated in place.
 *   q_new   bf16 [n_new][d].
 *   forced  NULL, or [events_cap][b_min] picks dictated to the compressions
 *           (-1: the argmin), passed to bkvo_fps_adopt (test harness only).
 *   ev_*    if not NULL, receive for each compression (events_cap at most) its
 *           b_min picks (indices into the full buffer), gaps, runner-up rows,
 *           margins and candidate values ([b_min][b_max] per compression), as
 *           bkvo_fps_adopt reports them.
 * Returns the number of compressions, or -1 if a forced pick was invalid.
 */
int bkvo_cfps_update(uint16_t* buf, int32_t* size, int b_min, int b_max, const uint16_t* q_new, int n_new, int d,
                     const int32_t* forced, int32_t* ev_picks, double* ev_gaps, int32_t* ev_alts, double* ev_margins,
                     double* ev_vals, int events_cap) {
  int n_ev = 0, bad = 0;
  const size_t nm = (size_t)(b_min > 0 ? b_min : 1);
  int32_t* picks = (int32_t*)malloc(sizeof(int32_t) * nm);
  double* gaps = (double*)malloc(sizeof(double) * nm);
  int32_t* alts = (int32_t*)malloc(sizeof(int32_t) * nm);
  double* margins = (double*)malloc(sizeof(double) * nm);
  double* vals = (double*)malloc(sizeof(double) * nm * (size_t)b_max);
  uint16_t* tmp = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)b_max * (size_t)d);
  for (int n = 0; n < n_new && !bad; ++n) {
    memcpy(buf + (size_t)(*size) * d, q_new + (size_t)n * d, sizeof(uint16_t) * (size_t)d);
    *size += 1;
    if (*size >= b_max) {
      const int32_t* f = (forced && n_ev < events_cap) ? forced + (size_t)n_ev * nm : NULL;
      int got = bkvo_fps_adopt(buf, *size, d, b_min, f, picks, gaps, alts, margins, vals);
      if (got < 0) {
        bad = 1;
        break;
      }
      for (int k = 0; k < got; ++k) memcpy(tmp + (size_t)k * d, buf + (size_t)picks[k] * d, sizeof(uint16_t) * (size_t)d);
      memcpy(buf, tmp, sizeof(uint16_t) * (size_t)got * (size_t)d);
      if (n_ev < events_cap) {
        if (ev_picks) memcpy(ev_picks + (size_t)n_ev * nm, picks, sizeof(int32_t) * (size_t)got);
        if (ev_gaps) memcpy(ev_gaps + (size_t)n_ev * nm, gaps, sizeof(double) * (size_t)got);
        if (ev_alts) memcpy(ev_alts + (size_t)n_ev * nm, alts, sizeof(int32_t) * (size_t)got);
        if (ev_margins) memcpy(ev_margins + (size_t)n_ev * nm, margins, sizeof(double) * (size_t)got);
        if (ev_vals) memcpy(ev_vals + (size_t)n_ev * nm * b_max, vals, sizeof(double) * (size_t)got * b_max);
      }
      ++n_ev;
      *size = got;
    }
  }
  free(tmp);
  free(vals);
  free(margins);
  free(alts);
  free(gaps);
  free(picks);
  return bad ? -1 : n_ev;
}

/* ------------------------------------------------------------------ */
/* Beacon state                                                        */
/* ------------------------------------------------------------------ */

/*
 * Prefill initialisation (Appendix D.2, Algorithm 2): FPS over the group's prompt queries
 * selects nb seeds; beacon k starts as the k-th pick with count 1.
 *   q: bf16 [N][d] (N = G * n_init, head-major); requires N >= nb.
 *   cent fp32 [nb][d], sums fp64 [nb][d], counts int64 [nb] are written.
 */
int bkvo_init_beacons(const uint16_t* q, int N, int d, int nb, float* cent, double* sums,
                      int64_t* counts, int32_t* picks, double* gap) {
  if (N < nb) return -1;
  int got = bkvo_fps(q, N, d, nb, picks, gap);
  for (int k = 0; k < got; ++k) {
    for (int i = 0; i < d; ++i) {
      double v = bkvo_bf16_to_f64(q[(size_t)picks[k] * d + i]);
      sums[(size_t)k * d + i] = v;
      cent[(size_t)k * d + i] = (float)v;
    }
    counts[k] = 1;
  }
  return got;
}

/*
 * One beacon-maintenance call: nearest-beacon assignment by cosine similarity
 * and a running-mean centroid update (the "K-Means Centroids" representative
 * the paper compares against Continual FPS in Section 4.2, Figure 7).
 *   Every query sees the centroids as they were when the call started.
 *   assign[n] = argmax over beacons b with count > 0 and |c_b| > 0 of
 *               cos(q_n, c_b); ties -> lowest b; -1 when |q_n| = 0 or no
 *               beacon qualifies.
 *   margin[n] = best cosine - runner-up cosine (+inf with one candidate).
 *   Then for every beacon b: sums_b += sum of its assigned queries (fp64, in
 *   row order), counts_b += their number, and if any arrived
 *   cent_b = fp32(sums_b / counts_b).
 * assign[] always reports the oracle's own argmax.  If override_assign is not
 * NULL, its entries decide which beacon each query is added to instead (the
 * parity tests use it to follow the GPU through exact ties).
 */
void bkvo_update(const uint16_t* q, int nq, int d, int nb, float* cent, double* sums, int64_t* counts,
                 const int32_t* override_assign, int32_t* assign, double* margin) {
  double* x = widen_rows(q, nq, d);
  double* c = (double*)malloc(sizeof(double) * (size_t)(nb > 0 ? nb : 1) * (size_t)d);
  char* ok = (char*)calloc((size_t)(nb > 0 ? nb : 1), 1);
  int32_t* chosen = (int32_t*)malloc(sizeof(int32_t) * (size_t)(nq > 0 ? nq : 1));
  for (int b = 0; b < nb; ++b) {
    for (int i = 0; i < d; ++i) c[(size_t)b * d + i] = (double)cent[(size_t)b * d + i];
    ok[b] = (counts[b] > 0 && dot_seq(c + (size_t)b * d, c + (size_t)b * d, d) > 0.0);
  }

  for (int n = 0; n < nq; ++n) {
    const double* qn = x + (size_t)n * d;
    int best_b = -1;
    double b1 = -INFINITY, b2 = -INFINITY;
    if (dot_seq(qn, qn, d) > 0.0) {
      for (int b = 0; b < nb; ++b) {
        if (!ok[b]) continue;
        double cs = cosine(qn, c + (size_t)b * d, d, NULL);
        if (cs > b1) {
          b2 = b1;
          b1 = cs;
          best_b = b;
        } else if (cs > b2) {
          b2 = cs;
        }
      }
    }
    if (assign) assign[n] = best_b;
    if (margin) margin[n] = (best_b >= 0 && b2 > -INFINITY) ? b1 - b2 : INFINITY;
    chosen[n] = override_assign ? override_assign[n] : best_b;
  }

  int64_t* add = (int64_t*)calloc((size_t)(nb > 0 ? nb : 1), sizeof(int64_t));
  for (int n = 0; n < nq; ++n) {
    int b = chosen[n];
    if (b < 0 || b >= nb) continue;
    for (int i = 0; i < d; ++i) sums[(size_t)b * d + i] = sums[(size_t)b * d + i] + x[(size_t)n * d + i];
    add[b] += 1;
  }
  for (int b = 0; b < nb; ++b) {
    if (add[b] == 0) continue;
    counts[b] += add[b];
    for (int i = 0; i < d; ++i)
      cent[(size_t)b * d + i] = (float)(sums[(size_t)b * d + i] / (double)counts[b]);
  }
  free(add);
  free(chosen);
  free(ok);
  free(c);
  free(x);
}

/* ------------------------------------------------------------------ */
/* Observation-query construction (Section 4.3; Appendix D.2)          */
/* ------------------------------------------------------------------ */

/* Rotary embedding of one vector at position pos, rotate-half pairing:
 *   a_i = pos * theta^(-2i/d),  i < d/2
 *   y_i       = x_i cos a_i - x_{i+d/2} sin a_i
 *   y_{i+d/2} = x_{i+d/2} cos a_i + x_i sin a_i
 * theta == 0 leaves x unchanged. */
void bkvo_rope(const double* x, int d, int64_t pos, double theta, double* y) {
  int h = d / 2;
  if (theta == 0.0) {
    for (int i = 0; i < d; ++i) y[i] = x[i];
    return;
  }
  for (int i = 0; i < h; ++i) {
    double inv_freq = pow(theta, -(double)(2 * i) / (double)d);
    double a = (double)pos * inv_freq;
    double cs = cos(a), sn = sin(a);
    double x1 = x[i], x2 = x[i + h];
    y[i] = x1 * cs - x2 * sn;
    y[i + h] = x2 * cs + x1 * sn;
  }
}

/*
 * Q_obs of one GQA group:
 *   rows [0, n_recent_rows)      recent queries, row h*W + w rotated at recent_pos[w]
 *   rows [n_recent_rows, +nb)    beacons (centroids) rotated at the current step t
 * Each rotated vector is rounded fp64 -> fp32 -> bf16 (the scoring precision).
 * valid[row] = 1 for every recent row and for beacons with count > 0.
 * Returns the row count M = n_recent_rows + nb.
 */
int bkvo_build_qobs(const float* cent, const int64_t* counts, int nb, const uint16_t* q_recent,
                    int G, int W, const int64_t* recent_pos, int64_t t_pos, int d, double theta,
                    double* qobs, int32_t* valid) {
  double* x = (double*)malloc(sizeof(double) * (size_t)d);
  double* y = (double*)malloc(sizeof(double) * (size_t)d);
  int row = 0;
  for (int h = 0; h < G; ++h) {
    for (int w = 0; w < W; ++w, ++row) {
      for (int i = 0; i < d; ++i) x[i] = bkvo_bf16_to_f64(q_recent[((size_t)h * W + w) * d + i]);
      bkvo_rope(x, d, recent_pos[w], theta, y);
      for (int i = 0; i < d; ++i) qobs[(size_t)row * d + i] = bkvo_round_scoring(y[i]);
      valid[row] = 1;
    }
  }
  for (int b = 0; b < nb; ++b, ++row) {
    for (int i = 0; i < d; ++i) x[i] = (double)cent[(size_t)b * d + i];
    bkvo_rope(x, d, t_pos, theta, y);
    for (int i = 0; i < d; ++i) qobs[(size_t)row * d + i] = bkvo_round_scoring(y[i]);
    valid[row] = counts[b] > 0 ? 1 : 0;
  }
  free(y);
  free(x);
  return row;
}

/* ------------------------------------------------------------------ */
/* Scoring (Eq. 4; Eq. 6 max or mean form; group of Section 4.3)     */
/* ------------------------------------------------------------------ */

/*
 * For every valid observation query q and every cached key j visible to it:
 *   logit_qj = (q . k_j) / sqrt(d)
 *   w_qj     = exp(logit_qj) / sum_l exp(logit_ql)      (softmax over the visible keys l)
 * Score[j]   = max over valid q of w_qj            (mean == 0, Eq. 6 max form)
 *            = (1 / #valid) * sum over valid q of w_qj   (mean != 0, Eq. 6 mean form)
 * Without positions (qpos == NULL) every key is visible to every query: the
 * softmax runs over all L cached keys (Eq. 4).  With positions, key j is
 * visible to query q only if kpos[j] <= qpos[q] (causal mask); a masked
 * weight is 0, and a valid query still counts in #valid.
 * The normaliser is evaluated as lse_q = m_q + log(sum_l exp(logit_ql - m_q)),
 * m_q = max_l logit_ql, so that exp does not overflow.
 * Score[j] = 0 for every j when no query is valid.
 */
void bkvo_score_mask(const double* qobs, const int32_t* valid, const int64_t* qpos, int M, const uint16_t* K,
                     const int64_t* kpos, int L, int d, int mean, double* score) {
  double* k = widen_rows(K, L, d);
  double* lg = (double*)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  double inv_sqrt_d = 1.0 / sqrt((double)d);
  int n_valid = 0;
  for (int j = 0; j < L; ++j) score[j] = 0.0;
  for (int q = 0; q < M; ++q) {
    if (!valid[q]) continue;
    ++n_valid;
    double m = -INFINITY;
    for (int j = 0; j < L; ++j) {
      if (qpos && kpos[j] > qpos[q]) {
        lg[j] = -INFINITY; /* masked: exp gives 0 below */
        continue;
      }
      lg[j] = dot_seq(qobs + (size_t)q * d, k + (size_t)j * d, d) * inv_sqrt_d;
      if (lg[j] > m) m = lg[j];
    }
    if (m == -INFINITY) continue; /* sees no key: every weight is 0 */
    double s = 0.0;
    for (int j = 0; j < L; ++j) s = s + exp(lg[j] - m);
    double lse = m + log(s);
    for (int j = 0; j < L; ++j) {
      double w = exp(lg[j] - lse);
      if (mean)
        score[j] = score[j] + w;
      else if (w > score[j])
        score[j] = w;
    }
  }
  if (mean && n_valid > 0)
    for (int j = 0; j < L; ++j) score[j] = score[j] / (double)n_valid;
  free(lg);
  free(k);
}

void bkvo_score_agg(const double* qobs, const int32_t* valid, int M, const uint16_t* K, int L, int d, int mean,
                    double* score) {
  bkvo_score_mask(qobs, valid, NULL, M, K, NULL, L, d, mean, score);
}

void bkvo_score(const double* qobs, const int32_t* valid, int M, const uint16_t* K, int L, int d,
                double* score) {
  bkvo_score_agg(qobs, valid, M, K, L, d, 0, score);
}

/* ------------------------------------------------------------------ */
/* Selection (Eq. 7; keep set and TopK of Algorithm 2)                 */
/* ------------------------------------------------------------------ */

typedef struct {
  double s;
  int32_t j;
} cand_t;

static int cand_cmp(const void* a, const void* b) {
  const cand_t* x = (const cand_t*)a;
  const cand_t* y = (const cand_t*)b;
  if (x->s > y->s) return -1;
  if (x->s < y->s) return 1;
  return (x->j < y->j) ? -1 : (x->j > y->j);
}

static int int_cmp(const void* a, const void* b) {
  int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
  return (x > y) - (x < y);
}

/*
 * I_keep = [0, n_prefix) U [L - W, L);  k_sel = budget - |I_keep|;
 * I_top  = the k_sel candidates outside I_keep with the largest Score,
 *          ordered by (Score descending, index ascending);
 * kept   = Sort(I_keep U I_top), ascending.
 * When L <= budget nothing is evicted and kept = 0 .. L-1.
 * boundary[0] = score of the last candidate taken, boundary[1] = score of the
 * first candidate left out (NaN where it does not exist).
 * Returns the number of kept indices, or -1 if budget < n_prefix + W.
 */
int bkvo_select(const double* score, int L, int budget, int W, int n_prefix, int32_t* kept,
                double* boundary) {
  boundary[0] = NAN;
  boundary[1] = NAN;
  if (L <= budget) {
    for (int j = 0; j < L; ++j) kept[j] = j;
    return L;
  }
  if (budget < n_prefix + W) return -1;
  int n_keep = 0;
  for (int j = 0; j < n_prefix; ++j) kept[n_keep++] = j;
  for (int j = L - W; j < L; ++j) kept[n_keep++] = j;
  int k_sel = budget - n_keep;
  int nc = L - W - n_prefix;
  cand_t* c = (cand_t*)malloc(sizeof(cand_t) * (size_t)(nc > 0 ? nc : 1));
  for (int t = 0; t < nc; ++t) {
    c[t].j = n_prefix + t;
    c[t].s = score[n_prefix + t];
  }
  qsort(c, (size_t)nc, sizeof(cand_t), cand_cmp);
  for (int t = 0; t < k_sel; ++t) kept[n_keep++] = c[t].j;
  if (k_sel > 0) boundary[0] = c[k_sel - 1].s;
  if (k_sel < nc) boundary[1] = c[k_sel].s;
  qsort(kept, (size_t)n_keep, sizeof(int32_t), int_cmp);
  free(c);
  return n_keep;
}

/* ------------------------------------------------------------------ */
/* Gather / compaction (Eq. 8; Gather of Algorithm 2)                  */
/* ------------------------------------------------------------------ */

/* K_hat[i] = K[kept[i]], V_hat[i] = V[kept[i]] for i < n_kept, written back to
 * rows 0 .. n_kept-1 of the same buffers; rows >= n_kept are left as they were. */
void bkvo_gather(uint16_t* K, uint16_t* V, const int32_t* kept, int n_kept, int d) {
  size_t row = (size_t)d * sizeof(uint16_t);
  uint16_t* tk = (uint16_t*)malloc(row * (size_t)(n_kept > 0 ? n_kept : 1));
  uint16_t* tv = (uint16_t*)malloc(row * (size_t)(n_kept > 0 ? n_kept : 1));
  for (int i = 0; i < n_kept; ++i) {
    memcpy(tk + (size_t)i * d, K + (size_t)kept[i] * d, row);
    memcpy(tv + (size_t)i * d, V + (size_t)kept[i] * d, row);
  }
  memcpy(K, tk, row * (size_t)n_kept);
  memcpy(V, tv, row * (size_t)n_kept);
  free(tv);
  free(tk);
}

/* ------------------------------------------------------------------ */
/* Whole step over many instances (the CPU baseline, OpenMP)           */
/* ------------------------------------------------------------------ */

/*
 * Runs, for each listed instance, one beacon-maintenance call followed by one
 * compression, exactly as the per-instance functions above define them.
 * Layouts are those of the C-ABI (row-major):
 *   q_new    bf16 [n_inst_total][G][n_new][d]   (query heads of a group are adjacent)
 *   q_recent bf16 [n_inst_total][G][W][d]
 *   K, V     bf16 [n_inst_total][cap][d]        (modified in place)
 *   cent fp32 [n_inst_total][nb][d], sums fp64 [..][nb][d], counts int64 [..][nb]
 *   kept     int32 [n_inst_total][budget]
 *   score    fp64 [n_inst_total][cap] (may be NULL)
 * inst[] lists the instances to process (n_list of them).
 * Returns the number of OpenMP threads used.
 */
int bkvo_step_many(const int64_t* inst, int n_list, int G, int d, int nb, int W, int n_prefix, int cap,
                   const uint16_t* q_new, int n_new, const uint16_t* q_recent, const int64_t* recent_pos,
                   int64_t t_pos, double theta, int L, int budget, uint16_t* K, uint16_t* V, float* cent,
                   double* sums, int64_t* counts, int32_t* kept, double* score) {
  int threads = 1;
#ifdef _OPENMP
#pragma omp parallel
  {
#pragma omp single
    threads = omp_get_num_threads();
  }
#pragma omp parallel for schedule(dynamic, 1)
#endif
  for (int t = 0; t < n_list; ++t) {
    int64_t e = inst[t];
    int M = G * W + nb;
    if (n_new > 0)
      bkvo_update(q_new + (size_t)e * G * n_new * d, G * n_new, d, nb, cent + (size_t)e * nb * d,
                  sums + (size_t)e * nb * d, counts + (size_t)e * nb, NULL, NULL, NULL);
    double* qo = (double*)malloc(sizeof(double) * (size_t)M * d);
    int32_t* va = (int32_t*)malloc(sizeof(int32_t) * (size_t)M);
    double* sc = (double*)malloc(sizeof(double) * (size_t)L);
    int32_t* kp = (int32_t*)malloc(sizeof(int32_t) * (size_t)(L > budget ? budget : L));
    double bd[2];
    bkvo_build_qobs(cent + (size_t)e * nb * d, counts + (size_t)e * nb, nb, q_recent + (size_t)e * G * W * d,
                    G, W, recent_pos, t_pos, d, theta, qo, va);
    bkvo_score(qo, va, M, K + (size_t)e * cap * d, L, d, sc);
    int nk = bkvo_select(sc, L, budget, W, n_prefix, kp, bd);
    if (nk > 0) {
      bkvo_gather(K + (size_t)e * cap * d, V + (size_t)e * cap * d, kp, nk, d);
      memcpy(kept + (size_t)e * budget, kp, sizeof(int32_t) * (size_t)nk);
    }
    if (score) memcpy(score + (size_t)e * cap, sc, sizeof(double) * (size_t)L);
    free(kp);
    free(sc);
    free(va);
    free(qo);
  }
  return threads;
}
