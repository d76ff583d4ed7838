/*
 * CPU oracle for the GBA aggregate-and-apply step (arXiv 2205.11048).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, plain, single-threaded
 * statement of what one global step of GBA computes on the parameter server.
 * Only the tests, the smoke check and the benchmark's CPU-baseline leg may
 * load it.  The GPU library shares no code, header or table with it.
 *
 * Numerics: every gradient sum is accumulated in double and rounded once to
 * float; every other operation (division by the denominator, the optimizer
 * update) is done in float, one IEEE operation at a time, in the order written
 * below.  Build with -ffp-contract=off so no multiply-add is fused.
 *
 * What each part follows:
 *   - message weights f = [k - token <= iota]       Sec. 4.1, Eq. (1)
 *   - dense: weighted sum over the popped gradients divided by N_a
 *                                                   Alg. 2 (push responding)
 *   - embeddings: per-ID step tags, decay by tag vs token, weighted sum divided
 *     by the number of workers whose batches contained the ID
 *                                                   Alg. 2 (push responding)
 *   - update form w <- w - eta * v, v = (1/M) sum g  Appendix A, proof of Thm 1
 *   - optimizers Adagrad / Adam                      Table 1
 * Readings where the paper is silent are stated next to the code that takes
 * them (negative staleness clamps to 0; rows with no kept gradient are left
 * untouched; per-ID tags are read before this step updates them).
 *
 * Parity pins: see tests/test_oracle_pins.py (hand-worked exact example,
 * zero-staleness closed form against a linear-algebra statement of the
 * synchronous global batch, decay boundaries, order invariance, brute force,
 * textbook optimizers, SplitMix64 published outputs).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define GBAO_ADAGRAD 0
#define GBAO_ADAM 1

typedef struct {
  int32_t kind;     /* GBAO_ADAGRAD or GBAO_ADAM */
  float lr;
  float init_acc;   /* Adagrad initial accumulator */
  float beta1, beta2, eps;
} gbao_opt;

/* One embedding table, restricted to a sorted set of tracked rows.  Rows are
 * independent of one another given the messages, so a tracked subset evolves
 * exactly as it would inside the full table. */
typedef struct {
  int64_t V;              /* rows in the table */
  int32_t d;              /* row width */
  int32_t id_mode;        /* 0: row = id (0 <= id < V), 1: row = (uint64)id mod V,
                             2: every distinct id is its own row (a hash table of
                                ids); the tracked "rows" are then ids */
  gbao_opt opt;
  int64_t n_track;        /* number of tracked rows */
  const int64_t* track;   /* tracked rows, strictly increasing (ids in id_mode 2) */
  float* w;               /* [n_track * d] */
  float* s0;              /* Adagrad accumulator or Adam first moment */
  float* s1;              /* Adam second moment (unused for Adagrad) */
  int64_t* ver;           /* per-ID step tag: global version after the last update */
} gbao_table;

/* Dense parameters, restricted to a tracked set of element indices. */
typedef struct {
  int64_t D;
  gbao_opt opt;
  int64_t n_track;
  const int64_t* track;   /* element indices in [0, D) */
  float* w;
  float* s0;
  float* s1;
} gbao_dense;

typedef struct {
  int32_t iota;                /* tolerance threshold of Eq. (1); INT32_MAX = keep all */
  int32_t row_staleness;       /* 0: tag of the ID vs token, 1: k vs token */
  int32_t sparse_denominator;  /* 0: messages that contain the ID, 1: kept ones, 2: M */
  int32_t decay;               /* 0: Eq. (1) as printed (weight 1 or 0);
                                  1: a kept gradient of staleness s weighs lambda^s */
  float lambda;                /* decay 1 only: 0 < lambda <= 1 */
  int32_t drop_latest;         /* Hop-BW backup workers: the last drop_latest popped
                                  gradients of a step are ignored (0: none) */
} gbao_rule;

/* Counters of one step (Table 3 reports dropped batches and staleness). */
typedef struct {
  int64_t msgs_kept, msgs_dropped;
  int64_t dense_stale_sum, dense_stale_max;
  int64_t pairs, pairs_dropped;         /* distinct (message, row) pairs seen */
  int64_t row_stale_sum, row_stale_max; /* over those pairs */
  int64_t occurrences;                  /* id occurrences whose row is tracked */
  int64_t rows_touched, rows_applied;
} gbao_stats;

/* ------------------------------------------------------------------ */
/* SplitMix64 (Steele, Lea, Flood 2014): the output for state x is the  */
/* mix of x + golden gamma.                                            */
/* ------------------------------------------------------------------ */
uint64_t gbao_splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

/* Initial weight of element e of the array tagged `tag`: the top 24 bits of
 * the hash, centred and scaled by 2^-27, so the value is an exact float in
 * [-1/16, 1/16). */
float gbao_init_weight(uint64_t seed, uint64_t tag, uint64_t e) {
  uint64_t h = gbao_splitmix64(seed ^ tag ^ e);
  int32_t top = (int32_t)(h >> 40) - 8388608;
  return (float)top * 0x1p-27f;
}

uint64_t gbao_table_tag(int32_t t) { return ((uint64_t)(uint32_t)t + 1u) << 48; }
uint64_t gbao_dense_tag(void) { return (uint64_t)0xFFFFu << 48; }

/* Fill the state of the tracked rows / elements with their initial values. */
void gbao_init_table(gbao_table* tb, int32_t t, uint64_t seed) {
  for (int64_t r = 0; r < tb->n_track; ++r) {
    for (int32_t j = 0; j < tb->d; ++j) {
      uint64_t e = (uint64_t)tb->track[r] * (uint64_t)tb->d + (uint64_t)j;
      int64_t i = r * tb->d + j;
      tb->w[i] = gbao_init_weight(seed, gbao_table_tag(t), e);
      if (tb->opt.kind == GBAO_ADAGRAD) {
        tb->s0[i] = tb->opt.init_acc;
      } else {
        tb->s0[i] = 0.0f;
        tb->s1[i] = 0.0f;
      }
    }
    tb->ver[r] = 0;
  }
}

void gbao_init_dense(gbao_dense* dn, uint64_t seed) {
  for (int64_t r = 0; r < dn->n_track; ++r) {
    uint64_t e = (uint64_t)dn->track[r];
    dn->w[r] = gbao_init_weight(seed, gbao_dense_tag(), e);
    if (dn->opt.kind == GBAO_ADAGRAD) {
      dn->s0[r] = dn->opt.init_acc;
    } else {
      dn->s0[r] = 0.0f;
      dn->s1[r] = 0.0f;
    }
  }
}

/* ------------------------------------------------------------------ */
/* Optimizers (Table 1 names them; the formulas are the textbook ones). */
/* ------------------------------------------------------------------ */

/* Adam bias corrections for step t = k + 1: beta^t as t successive double
 * multiplications, then 1 - beta^t rounded to float. */
static float adam_bias_correction(float beta, int64_t t) {
  double p = 1.0;
  for (int64_t i = 0; i < t; ++i) p = p * (double)beta;
  return (float)(1.0 - p);
}

/* Adagrad (Duchi, Hazan, Singer 2011): a <- a + g*g; w <- w - lr*g / sqrt(a). */
static void adagrad_update(const gbao_opt* o, float* w, float* a, float g) {
  float gg = g * g;
  float an = *a + gg;
  float step = o->lr * g;
  float den = sqrtf(an);
  *a = an;
  *w = *w - step / den;
}

/* Adam (Kingma, Ba 2015):
 * m <- b1*m + (1-b1)*g; v <- b2*v + (1-b2)*g*g;
 * w <- w - lr*(m/bc1) / (sqrt(v/bc2) + eps). */
static void adam_update(const gbao_opt* o, float* w, float* m, float* v, float g,
                        float bc1, float bc2) {
  float c1 = 1.0f - o->beta1;
  float c2 = 1.0f - o->beta2;
  float mn = o->beta1 * *m + c1 * g;
  float gg = g * g;
  float vn = o->beta2 * *v + c2 * gg;
  float mhat = mn / bc1;
  float vhat = vn / bc2;
  float num = o->lr * mhat;
  float den = sqrtf(vhat) + o->eps;
  *m = mn;
  *v = vn;
  *w = *w - num / den;
}

static void apply_opt(const gbao_opt* o, float* w, float* s0, float* s1, float g,
                      float bc1, float bc2) {
  if (o->kind == GBAO_ADAGRAD)
    adagrad_update(o, w, s0, g);
  else
    adam_update(o, w, s0, s1, g, bc1, bc2);
}

/* Position of row x among the tracked rows, or -1. */
static int64_t find_tracked(const int64_t* track, int64_t n, int64_t x) {
  int64_t lo = 0, hi = n;
  while (lo < hi) {
    int64_t mid = lo + (hi - lo) / 2;
    if (track[mid] < x)
      lo = mid + 1;
    else
      hi = mid;
  }
  return (lo < n && track[lo] == x) ? lo : -1;
}

/* Staleness of Eq. (1) with a token ahead of the reference clamped to 0. */
static int64_t staleness(int64_t ref, int64_t token) {
  int64_t s = ref - token;
  return s < 0 ? 0 : s;
}

/* The weight of a gradient with staleness s from the m-th popped message of
 * M.  Eq. (1): 0 beyond iota, else 1.  Sec. 4.1 leaves room for other decay
 * strategies; decay 1 weighs a kept gradient by lambda^s (s successive
 * multiplications in double, rounded once to float).  Sec. 5.1's Hop-BW
 * ignores the gradients of the slowest workers: with drop_latest = b3 the
 * last b3 popped messages weigh 0. */
static float decay_weight(const gbao_rule* rule, int64_t s, int32_t m, int32_t M) {
  if (s > (int64_t)rule->iota) return 0.0f;
  if (m >= M - rule->drop_latest) return 0.0f;
  if (rule->decay == 0) return 1.0f;
  double p = 1.0;
  for (int64_t i = 0; i < s; ++i) p = p * (double)rule->lambda;
  return (float)p;
}

/*
 * One global step k over the M popped messages.
 *
 * tokens[m]            token of message m
 * ids[t*M + m]         ids of message m for table t (n[t*M + m] of them)
 * rows[t*M + m]        their gradient rows, n * d floats, row-major
 * dense_grads[m]       dense gradient of message m, D floats
 * keep_msg_out[m]      (optional) f of Eq. (1) for message m
 * row_count_out[t]     (optional) per tracked row: messages containing it
 * row_kept_out[t]      (optional) per tracked row: kept occurrences
 *
 * Returns 0, or 1 when an id is out of range for a table in id_mode 0 or is
 * the reserved id INT64_MIN in id_mode 2.
 */
int gbao_step(int64_t k, const gbao_rule* rule, int32_t M, const int64_t* tokens,
              int32_t T, gbao_table* tables, const int64_t* const* ids,
              const int64_t* n, const float* const* rows, gbao_dense* dense,
              const float* const* dense_grads, int32_t* keep_msg_out,
              int64_t* const* row_count_out, int64_t* const* row_kept_out,
              gbao_stats* stats) {
  gbao_stats st;
  memset(&st, 0, sizeof st);

  /* Eq. (1): f(tau(m,k), k) = 0 if k - tau > iota, else 1 (or the weight of
   * the chosen decay strategy). */
  float* f = (float*)malloc(sizeof(float) * (size_t)(M > 0 ? M : 1));
  for (int32_t m = 0; m < M; ++m) {
    int64_t s = staleness(k, tokens[m]);
    f[m] = decay_weight(rule, s, m, M);
    if (f[m] > 0.0f) st.msgs_kept++; else st.msgs_dropped++;
    st.dense_stale_sum += s;
    if (s > st.dense_stale_max) st.dense_stale_max = s;
    if (keep_msg_out) keep_msg_out[m] = f[m] > 0.0f ? 1 : 0;
  }

  /* Adam bias corrections use the global step count t = k + 1. */
  int64_t t_step = k + 1;

  /* Dense: weighted sum of the popped gradients, divided by N_a (= M).  The
   * dense parameters take a step every global step, even when every message
   * was dropped (then the gradient is zero). */
  if (dense && dense->n_track > 0) {
    float bc1 = 1.0f, bc2 = 1.0f;
    if (dense->opt.kind == GBAO_ADAM) {
      bc1 = adam_bias_correction(dense->opt.beta1, t_step);
      bc2 = adam_bias_correction(dense->opt.beta2, t_step);
    }
    for (int64_t r = 0; r < dense->n_track; ++r) {
      int64_t e = dense->track[r];
      double S = 0.0;
      for (int32_t m = 0; m < M; ++m)
        if (f[m] > 0.0f) S += (double)f[m] * (double)dense_grads[m][e];
      float gsum = (float)S;
      float g = gsum / (float)M;
      apply_opt(&dense->opt, &dense->w[r], &dense->s0[r],
                dense->s1 ? &dense->s1[r] : NULL, g, bc1, bc2);
    }
  }

  int err = 0;
  for (int32_t t = 0; t < T; ++t) {
    gbao_table* tb = &tables[t];
    int64_t nt = tb->n_track;
    int32_t d = tb->d;
    double* S = (double*)calloc((size_t)(nt > 0 ? nt : 1) * (size_t)d, sizeof(double));
    int64_t* cnt = (int64_t*)calloc((size_t)(nt > 0 ? nt : 1), sizeof(int64_t));
    int64_t* cnt_kept = (int64_t*)calloc((size_t)(nt > 0 ? nt : 1), sizeof(int64_t));
    int64_t* kept_occ = (int64_t*)calloc((size_t)(nt > 0 ? nt : 1), sizeof(int64_t));
    int64_t* last_m = (int64_t*)malloc(sizeof(int64_t) * (size_t)(nt > 0 ? nt : 1));
    for (int64_t r = 0; r < nt; ++r) last_m[r] = -1;

    /* Decay each embedding gradient by the tag of its ID and the token.  The
     * tags are read here, before this step updates any of them. */
    for (int32_t m = 0; m < M; ++m) {
      const int64_t* idm = ids[(int64_t)t * M + m];
      const float* gm = rows[(int64_t)t * M + m];
      int64_t nm = n[(int64_t)t * M + m];
      for (int64_t i = 0; i < nm; ++i) {
        int64_t id = idm[i];
        int64_t x;
        if (tb->id_mode == 0) {
          if (id < 0 || id >= tb->V) { err = 1; continue; }
          x = id;
        } else if (tb->id_mode == 1) {
          x = (int64_t)((uint64_t)id % (uint64_t)tb->V);
        } else {
          if (id == INT64_MIN) { err = 1; continue; }  /* the reserved id */
          x = id;
        }
        int64_t r = find_tracked(tb->track, nt, x);
        if (r < 0) continue;
        st.occurrences++;
        int64_t ref = (rule->row_staleness == 0) ? tb->ver[r] : k;
        int64_t s = staleness(ref, tokens[m]);
        float fo = decay_weight(rule, s, m, M);
        int keep = fo > 0.0f;
        if (last_m[r] != m) {   /* first time row x is met in message m */
          last_m[r] = m;
          cnt[r]++;
          st.pairs++;
          st.row_stale_sum += s;
          if (s > st.row_stale_max) st.row_stale_max = s;
          if (keep) cnt_kept[r]++; else st.pairs_dropped++;
        }
        if (keep) {
          kept_occ[r]++;
          for (int32_t j = 0; j < d; ++j) S[r * d + j] += (double)fo * (double)gm[i * d + j];
        }
      }
    }

    float bc1 = 1.0f, bc2 = 1.0f;
    if (tb->opt.kind == GBAO_ADAM) {
      bc1 = adam_bias_correction(tb->opt.beta1, t_step);
      bc2 = adam_bias_correction(tb->opt.beta2, t_step);
    }
    /* Weighted sum divided by the number of workers whose batches contained the ID;
     * rows whose gradients were all excluded take no step and keep their tag. */
    for (int64_t r = 0; r < nt; ++r) {
      if (cnt[r] > 0) st.rows_touched++;
      if (row_count_out && row_count_out[t]) row_count_out[t][r] = cnt[r];
      if (row_kept_out && row_kept_out[t]) row_kept_out[t][r] = kept_occ[r];
      if (kept_occ[r] == 0) continue;
      int64_t denom = cnt[r];
      if (rule->sparse_denominator == 1) denom = cnt_kept[r];
      if (rule->sparse_denominator == 2) denom = M;
      for (int32_t j = 0; j < d; ++j) {
        float gsum = (float)S[r * d + j];
        float g = gsum / (float)denom;
        int64_t i = r * d + j;
        apply_opt(&tb->opt, &tb->w[i], &tb->s0[i], tb->s1 ? &tb->s1[i] : NULL, g, bc1,
                  bc2);
      }
      tb->ver[r] = k + 1;
      st.rows_applied++;
    }
    free(S);
    free(cnt);
    free(cnt_kept);
    free(kept_occ);
    free(last_m);
  }
  free(f);
  if (stats) *stats = st;
  return err;
}

/* The paper's trigger: apply once at least the global batch is buffered, and
 * pop the oldest messages.  With local batches B[0..n) in arrival order this
 * returns the length of the shortest prefix whose total reaches G, or 0. */
int32_t gbao_select_prefix(const int32_t* B, int32_t n, int64_t G) {
  int64_t acc = 0;
  for (int32_t i = 0; i < n; ++i) {
    acc += B[i];
    if (acc >= G) return i + 1;
  }
  return 0;
}
