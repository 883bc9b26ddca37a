/*
 * oracle.c -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, single-threaded fp64 CPU statement of what the bucketed
 * LSTM-CTC training step computes.  Only the test suite, the smoke check and
 * the benchmark's CPU-baseline leg may load this file's library; the product
 * path (the CUDA library) never does, and shares no code with it.
 *
 * Contents, each following the passage named beside it:
 *   or_splitmix64       SplitMix64 (Steele, Lea & Flood, "Fast splittable
 *                       pseudorandom number generators", OOPSLA 2014).  The
 *                       paper names no generator; this is the shuffle source.
 *   or_histogram        Section III.A: f[l] = number of sequences of length l.
 *   or_dynamic_bucketing  Section III.A, procedure DYNAMICBUCKETING: the
 *                       dynamic program over the length histogram, in the
 *                       paper's loop order (q, then i, then j descending) with
 *                       the strict "<" update, then the back-pointer walk.
 *   or_plan             Section III.A/B and IV.A: assign each sequence to the
 *                       first bucket whose upper bound holds its length,
 *                       shuffle inside each bucket, cut mini-batches, emit the
 *                       buckets shortest first.
 *   or_plan_ordered     the same plan with the batches emitted in another
 *                       order (Section V leaves bucket-ordering strategies to
 *                       future work): descending buckets, a shuffled bucket
 *                       sequence, or all batches shuffled.
 *   or_ctc              CTC (Graves et al. 2006, the paper's ref. [15]):
 *                       log-space forward/backward variables and the gradient
 *                       of -ln p with respect to the unnormalised outputs.
 *   or_lstm_ctc_step    The training step: stacked (bi)directional LSTM
 *                       (Hochreiter & Schmidhuber, ref. [1]; gates i, f, g, o,
 *                       no peepholes), linear output + log-softmax, CTC loss,
 *                       and exact back-propagation through time.  Every
 *                       sequence is processed alone over its own length, so no
 *                       padding ever enters the arithmetic (eq. 1-2 are the
 *                       padded cost this removes).
 *   or_sgd              theta <- theta - lr * g.
 *   or_adadelta         ADADELTA (Zeiler 2012, the paper's ref. [21], its
 *                       Algorithm 1), the update rule of Section III.B step 4.
 *   or_average_models   Section III.B step 5, eq. 3 with alpha = 1: the main
 *                       process averages the parallel models' parameters and
 *                       subtracts beta times the previous epoch's values.
 *
 * Numerics: all arithmetic is in double; exp/log/tanh are the C library's.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_EINVAL 1
#define OR_ENOMEM 2

/* "INF" of the dynamic program (Section III.A notation list). */
#define OR_DP_INF ((int64_t)1 << 62)

/* ------------------------------------------------------------------ */
/* SplitMix64: state advances by the golden-ratio increment, then the
 * output is the variant-13 finaliser of the new state.                */
uint64_t or_splitmix64(uint64_t *state) {
  uint64_t z;
  *state += 0x9E3779B97F4A7C15ULL;
  z = *state;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/* ------------------------------------------------------------------ */
/* Section III.A: "an array f that stores a number of sequences for each
 * length".  f has lmax+1 entries, indexed by the length itself.       */
int or_histogram(const int32_t *lengths, int64_t n, int32_t lmax, int64_t *f) {
  int64_t i;
  if (!lengths || !f || n < 1 || lmax < 1) return OR_EINVAL;
  for (i = 0; i <= lmax; i++) f[i] = 0;
  for (i = 0; i < n; i++) {
    if (lengths[i] < 1 || lengths[i] > lmax) return OR_EINVAL;
    f[lengths[i]] += 1;
  }
  return OR_OK;
}

/* ------------------------------------------------------------------ */
/* Section III.A, DYNAMICBUCKETING(Q, f).
 *   dp[q][i]   best cost of cutting lengths 1..i into q groups, each group
 *              charged (its upper length i) x (its sequence count);
 *   prev[q][i] where the (q-1)-th group ended in that best cut.
 * dp[0][0] = 0 and every other entry starts at INF.  The i loop runs over
 * 1..n-1 (n = length(f)): the walk back starts at n-1, and f[n] does not
 * exist.  The j loop runs from i-1 down to 0 and keeps the first strict
 * improvement, so among equal costs the largest j wins.
 * Output: bests[0..Q-1] = upper bounds b_1 < ... < b_Q = n-1, and the
 * optimal cost dp[Q][n-1].  Q > n-1 leaves dp[Q][n-1] at INF: EINVAL. */
int or_dynamic_bucketing(const int64_t *f, int32_t n, int32_t Q,
                         int32_t *bests, int64_t *cost) {
  int64_t *dp, *prev_dp;
  int32_t q, i, j, cur_id;
  if (!f || !bests || n < 2 || Q < 1) return OR_EINVAL;
  if (Q > n - 1) return OR_EINVAL;
  dp = (int64_t *)malloc(sizeof(int64_t) * (size_t)(Q + 1) * (size_t)n);
  prev_dp = (int64_t *)malloc(sizeof(int64_t) * (size_t)(Q + 1) * (size_t)n);
  if (!dp || !prev_dp) {
    free(dp);
    free(prev_dp);
    return OR_ENOMEM;
  }
  for (i = 0; i < (Q + 1) * n; i++) {
    dp[i] = OR_DP_INF;
    prev_dp[i] = -1;
  }
  dp[0] = 0; /* dp[0][0] */
  for (q = 1; q <= Q; q++) {
    for (i = 1; i <= n - 1; i++) {
      int64_t cur_sum = f[i];
      for (j = i - 1; j >= 0; j--) {
        int64_t val = cur_sum * (int64_t)i + dp[(size_t)(q - 1) * n + j];
        if (val < dp[(size_t)q * n + i]) {
          dp[(size_t)q * n + i] = val;
          prev_dp[(size_t)q * n + i] = j;
        }
        cur_sum += f[j];
      }
    }
  }
  if (dp[(size_t)Q * n + (n - 1)] >= OR_DP_INF) {
    free(dp);
    free(prev_dp);
    return OR_EINVAL;
  }
  if (cost) *cost = dp[(size_t)Q * n + (n - 1)];
  cur_id = n - 1;
  for (q = Q; q >= 1; q--) {
    bests[q - 1] = cur_id; /* push_front */
    cur_id = (int32_t)prev_dp[(size_t)q * n + cur_id];
  }
  free(dp);
  free(prev_dp);
  return OR_OK;
}

/* ------------------------------------------------------------------ */
/* The epoch plan.
 *   1. f from the lengths, lmax = the largest length; the DP gives bounds.
 *   2. bucket(s) = the smallest q with L_s <= b_q.  Each bucket lists its
 *      sequences in ascending original index.
 *   3. One SplitMix64 stream, state0 = seed + (epoch+1) * 0x9E3779B97F4A7C15
 *      (mod 2^64), walks the buckets in ascending q; inside a bucket of m
 *      entries a Fisher-Yates pass runs k = m-1 .. 1 with j = next() mod
 *      (k+1), then swaps entries k and j.
 *   4. order = the buckets concatenated, shortest bucket first (Section
 *      IV.A: the shorter sequences are fed first).  Each bucket is cut into
 *      consecutive mini-batches of `batch` entries; its last one may be
 *      partial and is kept.  batch_off[b]..batch_off[b+1] indexes order.
 *   5. (or_plan_ordered) mode 0 keeps that order; mode 1 emits the buckets
 *      longest first; mode 2 permutes the bucket sequence 0..Q-1 by
 *      Fisher-Yates (k = Q-1 .. 1, j = next() mod (k+1)) drawing on from
 *      the same stream; mode 3 permutes all batches (in the order of step
 *      4) the same way.  Batches stay whole; order is rewritten to match.
 * Capacities: bounds[Q], order[n], batch_off[n+1], batch_bucket[n].    */
int or_plan_ordered(const int32_t *lengths, int64_t n, int32_t Q,
                    int32_t batch, uint64_t seed, uint64_t epoch,
                    int32_t mode, int32_t *bounds, int64_t *dp_cost,
                    int32_t *order, int32_t *batch_off, int32_t *batch_bucket,
                    int32_t *n_batches, int64_t *padded_timesteps) {
  int32_t lmax = 0, q;
  int64_t i, *f, padded = 0;
  int32_t nb = 0;
  int32_t *bucket_of, *bucket_start, *bucket_fill;
  uint64_t state;
  int rc;
  if (!lengths || n < 1 || Q < 1 || batch < 1 || !bounds || !order ||
      !batch_off || !batch_bucket || !n_batches || mode < 0 || mode > 3)
    return OR_EINVAL;
  for (i = 0; i < n; i++) {
    if (lengths[i] < 1) return OR_EINVAL;
    if (lengths[i] > lmax) lmax = lengths[i];
  }
  f = (int64_t *)malloc(sizeof(int64_t) * (size_t)(lmax + 1));
  if (!f) return OR_ENOMEM;
  rc = or_histogram(lengths, n, lmax, f);
  if (rc == OR_OK) rc = or_dynamic_bucketing(f, lmax + 1, Q, bounds, dp_cost);
  free(f);
  if (rc != OR_OK) return rc;

  bucket_of = (int32_t *)malloc(sizeof(int32_t) * (size_t)n);
  bucket_start = (int32_t *)calloc((size_t)Q + 1, sizeof(int32_t));
  bucket_fill = (int32_t *)calloc((size_t)Q, sizeof(int32_t));
  if (!bucket_of || !bucket_start || !bucket_fill) {
    free(bucket_of);
    free(bucket_start);
    free(bucket_fill);
    return OR_ENOMEM;
  }
  for (i = 0; i < n; i++) {
    q = 0;
    while (lengths[i] > bounds[q]) q++;
    bucket_of[i] = q;
    bucket_start[q + 1] += 1;
  }
  for (q = 0; q < Q; q++) bucket_start[q + 1] += bucket_start[q];
  /* ascending original index inside each bucket */
  for (i = 0; i < n; i++) {
    q = bucket_of[i];
    order[bucket_start[q] + bucket_fill[q]] = (int32_t)i;
    bucket_fill[q] += 1;
  }
  state = seed + (epoch + 1ULL) * 0x9E3779B97F4A7C15ULL;
  for (q = 0; q < Q; q++) {
    int32_t *lst = order + bucket_start[q];
    int64_t m = bucket_start[q + 1] - bucket_start[q], k;
    for (k = m - 1; k >= 1; k--) {
      int64_t j = (int64_t)(or_splitmix64(&state) % (uint64_t)(k + 1));
      int32_t t = lst[k];
      lst[k] = lst[j];
      lst[j] = t;
    }
  }
  for (q = 0; q < Q; q++) {
    int64_t s;
    for (s = bucket_start[q]; s < bucket_start[q + 1]; s += batch) {
      int64_t e = s + batch, r;
      int32_t mx = 0;
      if (e > bucket_start[q + 1]) e = bucket_start[q + 1];
      batch_off[nb] = (int32_t)s;
      batch_bucket[nb] = q;
      for (r = s; r < e; r++)
        if (lengths[order[r]] > mx) mx = lengths[order[r]];
      padded += (e - s) * (int64_t)mx;
      nb++;
    }
  }
  batch_off[nb] = (int32_t)n;
  *n_batches = nb;
  if (padded_timesteps) *padded_timesteps = padded;
  free(bucket_of);
  free(bucket_start);
  free(bucket_fill);
  if (mode != 0) {
    /* The batches above are in ascending cut order.  seq lists them in
     * emission order; then order, batch_off and batch_bucket are rebuilt
     * from it. */
    int32_t *seq = (int32_t *)malloc(sizeof(int32_t) * (size_t)nb);
    int32_t *qseq = (int32_t *)malloc(sizeof(int32_t) * (size_t)Q);
    int32_t *old_order = (int32_t *)malloc(sizeof(int32_t) * (size_t)n);
    int32_t *old_off = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nb + 1));
    int32_t *old_bucket = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nb > 0 ? nb : 1));
    int32_t b, w = 0, k;
    if (!seq || !qseq || !old_order || !old_off || !old_bucket) {
      free(seq);
      free(qseq);
      free(old_order);
      free(old_off);
      free(old_bucket);
      return OR_ENOMEM;
    }
    memcpy(old_order, order, sizeof(int32_t) * (size_t)n);
    memcpy(old_off, batch_off, sizeof(int32_t) * (size_t)(nb + 1));
    if (nb > 0) memcpy(old_bucket, batch_bucket, sizeof(int32_t) * (size_t)nb);
    if (mode == 3) {
      /* every batch, shuffled by Fisher-Yates from the same stream */
      for (b = 0; b < nb; b++) seq[b] = b;
      for (k = nb - 1; k >= 1; k--) {
        int32_t j = (int32_t)(or_splitmix64(&state) % (uint64_t)(k + 1));
        int32_t t = seq[k];
        seq[k] = seq[j];
        seq[j] = t;
      }
    } else {
      /* a sequence of buckets, each bucket's batches in cut order */
      for (q = 0; q < Q; q++) qseq[q] = (mode == 1) ? Q - 1 - q : q;
      if (mode == 2) {
        for (k = Q - 1; k >= 1; k--) {
          int32_t j = (int32_t)(or_splitmix64(&state) % (uint64_t)(k + 1));
          int32_t t = qseq[k];
          qseq[k] = qseq[j];
          qseq[j] = t;
        }
      }
      for (q = 0; q < Q; q++)
        for (b = 0; b < nb; b++)
          if (old_bucket[b] == qseq[q]) seq[w++] = b;
    }
    w = 0;
    for (b = 0; b < nb; b++) {
      int32_t src = seq[b], r;
      batch_off[b] = w;
      batch_bucket[b] = old_bucket[src];
      for (r = old_off[src]; r < old_off[src + 1]; r++) order[w++] = old_order[r];
    }
    batch_off[nb] = (int32_t)n;
    free(seq);
    free(qseq);
    free(old_order);
    free(old_off);
    free(old_bucket);
  }
  return OR_OK;
}

int or_plan(const int32_t *lengths, int64_t n, int32_t Q, int32_t batch,
            uint64_t seed, uint64_t epoch, int32_t *bounds, int64_t *dp_cost,
            int32_t *order, int32_t *batch_off, int32_t *batch_bucket,
            int32_t *n_batches, int64_t *padded_timesteps) {
  return or_plan_ordered(lengths, n, Q, batch, seed, epoch, 0, bounds, dp_cost,
                         order, batch_off, batch_bucket, n_batches,
                         padded_timesteps);
}

/* ------------------------------------------------------------------ */
/* log(e^a + e^b) with -inf handled explicitly. */
static double lse2(double a, double b) {
  double m;
  if (a == -INFINITY) return b;
  if (b == -INFINITY) return a;
  m = a > b ? a : b;
  return m + log1p(exp(-fabs(a - b)));
}

/* CTC for one sequence (Graves et al. 2006, Sections 3.1-4.1).
 *   logp[T x C]: log-softmax outputs; labels[U], none equal to blank.
 *   Extended label l' (length S = 2U+1): blanks at even s, labels at odd s.
 *   alpha_t(s) includes the emission at t; beta_t(s) excludes it, so
 *   sum_s alpha_t(s) beta_t(s) = p for every t.
 *   Returns -ln p (+inf when no alignment exists, i.e. T < U + repeats).
 *   dlogit[T x C] (optional) receives d(-ln p)/d(unnormalised output)
 *   = softmax - sum_{s: l'_s = k} alpha_t(s) beta_t(s) / p, or all zeros
 *   when the sequence has no alignment.                               */
double or_ctc(const double *logp, int32_t T, int32_t C, int32_t blank,
              const int32_t *labels, int32_t U, double *dlogit) {
  int32_t S = 2 * U + 1, t, s, k;
  double *alpha, *beta, lnp;
  int32_t *ext;
  if (T < 1 || C < 1) return NAN;
  ext = (int32_t *)malloc(sizeof(int32_t) * (size_t)S);
  alpha = (double *)malloc(sizeof(double) * (size_t)T * S);
  beta = (double *)malloc(sizeof(double) * (size_t)T * S);
  if (!ext || !alpha || !beta) {
    free(ext);
    free(alpha);
    free(beta);
    return NAN;
  }
  for (s = 0; s < S; s++) ext[s] = (s % 2 == 0) ? blank : labels[(s - 1) / 2];
  for (s = 0; s < T * S; s++) {
    alpha[s] = -INFINITY;
    beta[s] = -INFINITY;
  }
  /* forward variables */
  alpha[0] = logp[blank];
  if (S > 1) alpha[1] = logp[ext[1]];
  for (t = 1; t < T; t++) {
    for (s = 0; s < S; s++) {
      double a = alpha[(size_t)(t - 1) * S + s];
      if (s >= 1) a = lse2(a, alpha[(size_t)(t - 1) * S + s - 1]);
      if (s >= 2 && ext[s] != blank && ext[s] != ext[s - 2])
        a = lse2(a, alpha[(size_t)(t - 1) * S + s - 2]);
      alpha[(size_t)t * S + s] =
          (a == -INFINITY) ? -INFINITY : a + logp[(size_t)t * C + ext[s]];
    }
  }
  lnp = alpha[(size_t)(T - 1) * S + S - 1];
  if (S > 1) lnp = lse2(lnp, alpha[(size_t)(T - 1) * S + S - 2]);
  if (lnp == -INFINITY) {
    if (dlogit) memset(dlogit, 0, sizeof(double) * (size_t)T * C);
    free(ext);
    free(alpha);
    free(beta);
    return INFINITY;
  }
  if (dlogit) {
    /* backward variables, emission at t excluded */
    beta[(size_t)(T - 1) * S + S - 1] = 0.0;
    if (S > 1) beta[(size_t)(T - 1) * S + S - 2] = 0.0;
    for (t = T - 2; t >= 0; t--) {
      for (s = 0; s < S; s++) {
        const double *bn = beta + (size_t)(t + 1) * S;
        const double *ln = logp + (size_t)(t + 1) * C;
        double b = -INFINITY;
        if (bn[s] != -INFINITY) b = bn[s] + ln[ext[s]];
        if (s + 1 < S && bn[s + 1] != -INFINITY)
          b = lse2(b, bn[s + 1] + ln[ext[s + 1]]);
        if (s + 2 < S && ext[s + 2] != blank && ext[s + 2] != ext[s] &&
            bn[s + 2] != -INFINITY)
          b = lse2(b, bn[s + 2] + ln[ext[s + 2]]);
        beta[(size_t)t * S + s] = b;
      }
    }
    for (t = 0; t < T; t++) {
      double *g = dlogit + (size_t)t * C;
      for (k = 0; k < C; k++) g[k] = exp(logp[(size_t)t * C + k]);
      for (s = 0; s < S; s++) {
        double ab = alpha[(size_t)t * S + s] + beta[(size_t)t * S + s];
        if (ab != -INFINITY) g[ext[s]] -= exp(ab - lnp);
      }
    }
  }
  free(ext);
  free(alpha);
  free(beta);
  return -lnp;
}

/* ------------------------------------------------------------------ */
/* Flat parameter layout (all row-major):
 *   for layer l = 0..L-1, for direction d = 0 (forward), 1 (reverse):
 *       W_ih [4H x D_l], W_hh [4H x H], b [4H]     gate blocks i, f, g, o
 *   then W_out [C x dirs*H], b_out [C].
 *   D_0 = in_dim, D_l = dirs*H for l > 0.                                */
int64_t or_param_count(int32_t n_layers, int32_t bidir, int32_t in_dim,
                       int32_t hidden, int32_t n_classes) {
  int64_t dirs = bidir ? 2 : 1, H = hidden, p = 0;
  int32_t l;
  for (l = 0; l < n_layers; l++) {
    int64_t D = (l == 0) ? in_dim : dirs * H;
    p += dirs * 4 * H * (D + H + 1);
  }
  p += (int64_t)n_classes * (dirs * H + 1);
  return p;
}

static double sigm(double x) { return 1.0 / (1.0 + exp(-x)); }

/* One sequence through the whole step.  Gradients are added into grads.
 * x[T x in_dim]; returns the CTC loss of the sequence.                  */
static double step_one(int32_t n_layers, int32_t dirs, int32_t in_dim,
                       int32_t H, int32_t C, int32_t blank, int32_t T,
                       const double *x, const int32_t *labels, int32_t U,
                       const double *params, double *grads, int *err) {
  /* per layer and direction: activated gates [T x 4H], cell [T x H],
   * hidden [T x H]; per layer: the layer output Y [T x dirs*H]         */
  size_t nld = (size_t)n_layers * dirs;
  double **gates = (double **)calloc(nld, sizeof(double *));
  double **cell = (double **)calloc(nld, sizeof(double *));
  double **Y = (double **)calloc((size_t)n_layers, sizeof(double *));
  double *logp = NULL, *dlogit = NULL, *dY = NULL, *dX = NULL;
  double loss = NAN;
  int32_t l, d, t, r, k, DH = dirs * H;
  size_t off;
  size_t *w_off = (size_t *)calloc(nld, sizeof(size_t));
  size_t out_off;
  *err = 0;
  if (!gates || !cell || !Y || !w_off) goto fail;
  off = 0;
  for (l = 0; l < n_layers; l++) {
    int32_t D = (l == 0) ? in_dim : DH;
    for (d = 0; d < dirs; d++) {
      w_off[(size_t)l * dirs + d] = off;
      off += (size_t)4 * H * (D + H + 1);
    }
  }
  out_off = off;
  for (l = 0; l < n_layers; l++) {
    Y[l] = (double *)calloc((size_t)T * DH, sizeof(double));
    if (!Y[l]) goto fail;
    for (d = 0; d < dirs; d++) {
      gates[(size_t)l * dirs + d] = (double *)calloc((size_t)T * 4 * H, sizeof(double));
      cell[(size_t)l * dirs + d] = (double *)calloc((size_t)T * H, sizeof(double));
      if (!gates[(size_t)l * dirs + d] || !cell[(size_t)l * dirs + d]) goto fail;
    }
  }
  logp = (double *)calloc((size_t)T * C, sizeof(double));
  dlogit = (double *)calloc((size_t)T * C, sizeof(double));
  dY = (double *)calloc((size_t)T * DH, sizeof(double));
  dX = (double *)calloc((size_t)T * DH, sizeof(double));
  if (!logp || !dlogit || !dY || !dX) goto fail;

  /* ---- forward: each layer, each direction over the sequence's own length */
  for (l = 0; l < n_layers; l++) {
    int32_t D = (l == 0) ? in_dim : DH;
    const double *X = (l == 0) ? x : Y[l - 1];
    for (d = 0; d < dirs; d++) {
      const double *Wih = params + w_off[(size_t)l * dirs + d];
      const double *Whh = Wih + (size_t)4 * H * D;
      const double *b = Whh + (size_t)4 * H * H;
      double *G = gates[(size_t)l * dirs + d], *Cc = cell[(size_t)l * dirs + d];
      int32_t step;
      for (step = 0; step < T; step++) {
        int32_t tt = (d == 0) ? step : T - 1 - step;    /* time index */
        int32_t tp = (d == 0) ? tt - 1 : tt + 1;        /* previous step */
        int has_prev = (step > 0);
        for (r = 0; r < 4 * H; r++) {
          double z = b[r];
          for (k = 0; k < D; k++) z += Wih[(size_t)r * D + k] * X[(size_t)tt * D + k];
          if (has_prev)
            for (k = 0; k < H; k++)
              z += Whh[(size_t)r * H + k] * Y[l][(size_t)tp * DH + d * H + k];
          G[(size_t)tt * 4 * H + r] = z;
        }
        for (k = 0; k < H; k++) {
          double *g = G + (size_t)tt * 4 * H;
          double ig = sigm(g[k]), fg = sigm(g[H + k]), gg = tanh(g[2 * H + k]),
                 og = sigm(g[3 * H + k]);
          double cprev = has_prev ? Cc[(size_t)tp * H + k] : 0.0;
          double cn = fg * cprev + ig * gg;
          g[k] = ig;
          g[H + k] = fg;
          g[2 * H + k] = gg;
          g[3 * H + k] = og;
          Cc[(size_t)tt * H + k] = cn;
          Y[l][(size_t)tt * DH + d * H + k] = og * tanh(cn);
        }
      }
    }
  }
  /* ---- output layer and log-softmax */
  {
    const double *Wout = params + out_off, *bout = Wout + (size_t)C * DH;
    for (t = 0; t < T; t++) {
      double mx = -INFINITY, se = 0.0;
      for (k = 0; k < C; k++) {
        double z = bout[k];
        for (r = 0; r < DH; r++) z += Wout[(size_t)k * DH + r] * Y[n_layers - 1][(size_t)t * DH + r];
        logp[(size_t)t * C + k] = z;
        if (z > mx) mx = z;
      }
      for (k = 0; k < C; k++) se += exp(logp[(size_t)t * C + k] - mx);
      for (k = 0; k < C; k++) logp[(size_t)t * C + k] -= mx + log(se);
    }
  }
  /* ---- CTC loss and its gradient w.r.t. the logits */
  for (k = 0; k < U; k++)
    if (labels[k] < 0 || labels[k] >= C || labels[k] == blank) *err = 1;
  if (*err) goto fail;
  loss = or_ctc(logp, T, C, blank, labels, U, dlogit);
  if (isinf(loss)) goto done; /* no alignment: contributes no gradient */

  /* ---- output layer backward */
  {
    const double *Wout = params + out_off;
    double *gWout = grads + out_off, *gbout = gWout + (size_t)C * DH;
    const double *Yt = Y[n_layers - 1];
    for (t = 0; t < T; t++) {
      for (k = 0; k < C; k++) {
        double gk = dlogit[(size_t)t * C + k];
        gbout[k] += gk;
        for (r = 0; r < DH; r++) {
          gWout[(size_t)k * DH + r] += gk * Yt[(size_t)t * DH + r];
          dY[(size_t)t * DH + r] += gk * Wout[(size_t)k * DH + r];
        }
      }
    }
  }
  /* ---- back-propagation through time, top layer first */
  for (l = n_layers - 1; l >= 0; l--) {
    int32_t D = (l == 0) ? in_dim : DH;
    const double *X = (l == 0) ? x : Y[l - 1];
    memset(dX, 0, sizeof(double) * (size_t)T * DH);
    for (d = 0; d < dirs; d++) {
      const double *Wih = params + w_off[(size_t)l * dirs + d];
      const double *Whh = Wih + (size_t)4 * H * D;
      double *gWih = grads + w_off[(size_t)l * dirs + d];
      double *gWhh = gWih + (size_t)4 * H * D;
      double *gb = gWhh + (size_t)4 * H * H;
      const double *G = gates[(size_t)l * dirs + d], *Cc = cell[(size_t)l * dirs + d];
      double *dh_next = (double *)calloc((size_t)H, sizeof(double));
      double *dc_next = (double *)calloc((size_t)H, sizeof(double));
      double *dz = (double *)calloc((size_t)4 * H, sizeof(double));
      int32_t step;
      if (!dh_next || !dc_next || !dz) {
        free(dh_next);
        free(dc_next);
        free(dz);
        goto fail;
      }
      for (step = T - 1; step >= 0; step--) {
        int32_t tt = (d == 0) ? step : T - 1 - step;
        int32_t tp = (d == 0) ? tt - 1 : tt + 1;
        int has_prev = (step > 0);
        const double *g = G + (size_t)tt * 4 * H;
        for (k = 0; k < H; k++) {
          double ig = g[k], fg = g[H + k], gg = g[2 * H + k], og = g[3 * H + k];
          double cn = Cc[(size_t)tt * H + k];
          double cprev = has_prev ? Cc[(size_t)tp * H + k] : 0.0;
          double tc = tanh(cn);
          double dh = dY[(size_t)tt * DH + d * H + k] + dh_next[k];
          double dc = dc_next[k] + dh * og * (1.0 - tc * tc);
          dz[k] = dc * gg * ig * (1.0 - ig);
          dz[H + k] = dc * cprev * fg * (1.0 - fg);
          dz[2 * H + k] = dc * ig * (1.0 - gg * gg);
          dz[3 * H + k] = dh * tc * og * (1.0 - og);
          dc_next[k] = dc * fg;
        }
        for (k = 0; k < H; k++) dh_next[k] = 0.0;
        for (r = 0; r < 4 * H; r++) {
          double zr = dz[r];
          gb[r] += zr;
          for (k = 0; k < D; k++) {
            gWih[(size_t)r * D + k] += zr * X[(size_t)tt * D + k];
            dX[(size_t)tt * DH + k] += zr * Wih[(size_t)r * D + k];
          }
          if (has_prev)
            for (k = 0; k < H; k++) {
              gWhh[(size_t)r * H + k] += zr * Y[l][(size_t)tp * DH + d * H + k];
              dh_next[k] += zr * Whh[(size_t)r * H + k];
            }
        }
      }
      free(dh_next);
      free(dc_next);
      free(dz);
    }
    if (l > 0) memcpy(dY, dX, sizeof(double) * (size_t)T * DH);
  }
done:
  goto cleanup;
fail:
  if (!*err) *err = 2;
  loss = NAN;
cleanup:
  if (gates)
    for (size_t i = 0; i < nld; i++) free(gates[i]);
  if (cell)
    for (size_t i = 0; i < nld; i++) free(cell[i]);
  if (Y)
    for (l = 0; l < n_layers; l++) free(Y[l]);
  free(gates);
  free(cell);
  free(Y);
  free(w_off);
  free(logp);
  free(dlogit);
  free(dY);
  free(dX);
  return loss;
}

/* The training step over a mini-batch.  x holds the sequences' feature rows
 * one sequence after another ([sum L x in_dim]); labels likewise.  grads is
 * overwritten with d(sum_i loss_i)/d(params); loss[i] = -ln p(z_i | x_i).
 * Sequences with no alignment get loss +inf and add no gradient.        */
int or_lstm_ctc_step(int32_t n_layers, int32_t bidir, int32_t in_dim,
                     int32_t hidden, int32_t n_classes, int32_t blank,
                     int32_t n_seq, const int32_t *lengths, const double *x,
                     const int32_t *label_lengths, const int32_t *labels,
                     const double *params, double *grads, double *loss) {
  int32_t i, dirs = bidir ? 2 : 1;
  int64_t P, xo = 0, lo = 0;
  if (n_layers < 1 || in_dim < 1 || hidden < 1 || n_classes < 2 || n_seq < 0 ||
      blank < 0 || blank >= n_classes || !params || !grads || !loss)
    return OR_EINVAL;
  P = or_param_count(n_layers, bidir, in_dim, hidden, n_classes);
  memset(grads, 0, sizeof(double) * (size_t)P);
  for (i = 0; i < n_seq; i++) {
    int err = 0;
    if (lengths[i] < 1 || label_lengths[i] < 0) return OR_EINVAL;
    loss[i] = step_one(n_layers, dirs, in_dim, hidden, n_classes, blank,
                       lengths[i], x + xo * in_dim, labels + lo,
                       label_lengths[i], params, grads, &err);
    if (err == 1) return OR_EINVAL;
    if (err) return OR_ENOMEM;
    xo += lengths[i];
    lo += label_lengths[i];
  }
  return OR_OK;
}

void or_sgd(double *params, const double *grads, int64_t n, double lr) {
  int64_t i;
  for (i = 0; i < n; i++) params[i] -= lr * grads[i];
}

/* ADADELTA, Zeiler 2012 (ref. [21]), Algorithm 1, one update for i < n:
 *   accumulate gradient:  E[g^2] <- rho E[g^2] + (1 - rho) g^2
 *   compute update:       dx = -(RMS[dx]_{t-1} / RMS[g]_t) g,
 *                         RMS[y] = sqrt(E[y^2] + eps)
 *   accumulate updates:   E[dx^2] <- rho E[dx^2] + (1 - rho) dx^2
 *   apply update:         x <- x + lr dx   (lr = 1 in the algorithm; a
 *                         learning-rate factor scales the applied step only)
 */
void or_adadelta(double *x, const double *g, double *eg2, double *edx2,
                 int64_t n, double rho, double eps, double lr) {
  int64_t i;
  for (i = 0; i < n; i++) {
    double rms_g, rms_dx, dx;
    eg2[i] = rho * eg2[i] + (1.0 - rho) * g[i] * g[i];
    rms_g = sqrt(eg2[i] + eps);
    rms_dx = sqrt(edx2[i] + eps);
    dx = -(rms_dx / rms_g) * g[i];
    edx2[i] = rho * edx2[i] + (1.0 - rho) * dx * dx;
    x[i] += lr * dx;
  }
}

/* Eq. 3 (Section III.B step 5, alpha = 1): V(t) = V_alpha(t) - beta V(t-1),
 * V_alpha(t) the mean over the K parallel models of their parameters after
 * the epoch, V(t-1) the parameters the epoch started from.
 *   models  [K][n], row k = model k;  prev [n];  out [n].               */
int or_average_models(const double *models, int32_t K, const double *prev, int64_t n, double beta,
                      double *out) {
  int64_t i;
  int32_t k;
  if (K < 1 || n < 0) return OR_EINVAL;
  for (i = 0; i < n; i++) {
    double s = 0.0;
    for (k = 0; k < K; k++) s += models[(int64_t)k * n + i];
    out[i] = s / (double)K - beta * prev[i];
  }
  return OR_OK;
}
