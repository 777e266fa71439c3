/*
 * topk_oracle.c -- plain, slow, fp64 CPU oracle for top-k attention.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may link, load or
 * call this file; only the tests, the package's smoke check and the CPU
 * baseline leg of the benchmark do.  It shares no code, header, table or
 * helper with the CUDA library.
 *
 * What it computes, per query row i of problem (b, h), written out from the
 * paper's definitions with no blocking, fusion or reordering:
 *
 *   Eq. 1  (dot-product attention, temperature folded into Q):
 *            s_ij = sum_t q_i[t] * k_j[t]
 *   Eq. 2  (masking): a key j is valid for query i unless B_ij = -inf.  The
 *          masks taken: causal (j <= i + Lk - Lq: the queries are the last
 *          Lq positions of the sequence, as when decoding against a cache of
 *          Lk keys), a key count per batch (j < kv_len[b]: key padding) and
 *          an arbitrary bit mask (bit j of query row i: 1 = valid).
 *   Eq. 4  (top-k attention): keep the k largest s_ij of row i, apply the
 *            activation to those k entries only, and weight the value rows:
 *            out_i = sum_{j in topk(i)} act(s_i, topk(i))_j * v_j
 *          act = softmax over the kept entries (attention), or
 *   Eq. 3  act = ReLU applied entry-wise (feed-forward layer cast as
 *          attention: Q = x, K = W1, V = W2, rows of W1/W2 are keys/values).
 *
 * Readings where the paper is silent (Sec. 2.2 gives none of these):
 *   - ties in s are broken toward the lower key index, i.e. the kept set is
 *     the first k entries of the total order (s descending, j ascending);
 *   - a row with fewer than k valid keys keeps all of them (k_eff = the
 *     number of valid keys), and the softmax covers those only; a row with
 *     no valid key outputs zeros;
 *   - top-k runs on the signed scores; ReLU is applied after selection.
 *
 * Arithmetic: inputs are widened exactly to double (bf16 by a 16-bit
 * shift; fp64 inputs, used by the finite-difference pins, are taken as
 * they are); all sums, the softmax and the weighted sum are in double.
 * Selection keeps a bounded heap of the k+1 best entries so that the
 * (k+1)-th score, which decides the near-tie rule, is reported too.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

#define ORACLE_F32 0
#define ORACLE_BF16 1
#define ORACLE_F64 2
#define ACT_SOFTMAX 0
#define ACT_RELU 1

static double widen(const void* base, size_t i, int dtype) {
  if (dtype == ORACLE_F32) return (double)((const float*)base)[i];
  if (dtype == ORACLE_F64) return ((const double*)base)[i];
  uint32_t bits = ((uint32_t)((const uint16_t*)base)[i]) << 16;
  float f;
  memcpy(&f, &bits, sizeof f);
  return (double)f;
}

typedef struct {
  double s;
  int32_t j;
} entry;

/* a ranks below b in the total order (s descending, j ascending) */
static int ranks_below(entry a, entry b) {
  return a.s < b.s || (a.s == b.s && a.j > b.j);
}

/* Min-heap keyed by rank: h[0] is the lowest-ranked entry kept. */
static void heap_sift_down(entry* h, int n, int p) {
  for (;;) {
    int c = 2 * p + 1;
    if (c >= n) return;
    if (c + 1 < n && ranks_below(h[c + 1], h[c])) c++;
    if (!ranks_below(h[c], h[p])) return;
    entry t = h[c];
    h[c] = h[p];
    h[p] = t;
    p = c;
  }
}

static void heap_sift_up(entry* h, int c) {
  while (c > 0) {
    int p = (c - 1) / 2;
    if (!ranks_below(h[c], h[p])) return;
    entry t = h[c];
    h[c] = h[p];
    h[p] = t;
    c = p;
  }
}

static int cmp_rank_desc(const void* a, const void* b) {
  const entry* x = (const entry*)a;
  const entry* y = (const entry*)b;
  if (ranks_below(*y, *x)) return -1;
  if (ranks_below(*x, *y)) return 1;
  return 0;
}

typedef struct {
  int act, dtype;
  const void *q, *k, *v;
  int64_t H, Lq, Lk, d, topk;
  int causal, vanilla;
  int64_t coff;            /* causal: key j is valid for query i iff j <= i + coff */
  const int32_t* kv_len;   /* [B] valid keys per batch, or NULL */
  const uint32_t* mask;    /* bit mask, or NULL: word (b*mbs + h*mhs + i*mw + j/32) */
  int64_t mbs, mhs, mw;
  const int64_t* rows;
  int64_t nrows;
  const int32_t* eval_idx; /* index-evaluate mode when non-NULL */
  double *out, *score, *next_score;
  int32_t* idx;
  int64_t begin, end;
  int status;
} job;

/* Eq. 2: is key j valid for query i of problem bh = b * H + h? */
static int key_valid(const job* J, int64_t bh, int64_t i, int64_t j) {
  const int64_t b = bh / J->H, h = bh % J->H;
  if (J->causal && j > i + J->coff) return 0;
  if (J->kv_len && j >= (int64_t)J->kv_len[b]) return 0;
  if (J->mask) {
    const uint32_t w = J->mask[b * J->mbs + h * J->mhs + i * J->mw + (j >> 5)];
    if (!((w >> (j & 31)) & 1u)) return 0;
  }
  return 1;
}

static double dot_row(const job* J, int64_t krow, const double* qbuf) {
  double acc = 0.0;
  for (int64_t t = 0; t < J->d; ++t) acc += qbuf[t] * widen(J->k, (size_t)(krow * J->d + t), J->dtype);
  return acc;
}

static void* run_rows(void* arg) {
  job* J = (job*)arg;
  const int64_t d = J->d, K = J->topk;
  double* qbuf = (double*)malloc(sizeof(double) * (size_t)d);
  entry* heap = (entry*)malloc(sizeof(entry) * (size_t)(K + 1 > 1 ? K + 1 : 1));
  entry* sel = (entry*)malloc(sizeof(entry) * (size_t)(J->Lk > K + 1 ? J->Lk : K + 1));
  double* w = (double*)malloc(sizeof(double) * (size_t)(J->Lk > K ? J->Lk : K));
  if (!qbuf || !heap || !sel || !w) {
    J->status = -1;
    goto done;
  }
  for (int64_t r = J->begin; r < J->end; ++r) {
    const int64_t row = J->rows ? J->rows[r] : r;
    const int64_t bh = row / J->Lq, i = row % J->Lq;
    for (int64_t t = 0; t < d; ++t) qbuf[t] = widen(J->q, (size_t)(row * d + t), J->dtype);
    int64_t nsel = 0;
    double next = -INFINITY;

    if (J->eval_idx) {
      /* index-evaluate: the kept set is given; recompute its scores. */
      for (int64_t t = 0; t < K; ++t) {
        int32_t j = J->eval_idx[r * K + t];
        if (j < 0) continue;
        if (j >= J->Lk) {
          J->status = -3;
          continue;
        }
        sel[nsel].j = j;
        sel[nsel].s = dot_row(J, bh * J->Lk + j, qbuf);
        nsel++;
      }
    } else if (J->vanilla) {
      /* Eq. 1 / Eq. 2: every valid key is kept. */
      for (int64_t j = 0; j < J->Lk; ++j) {
        if (!key_valid(J, bh, i, j)) continue;
        sel[nsel].j = (int32_t)j;
        sel[nsel].s = dot_row(J, bh * J->Lk + j, qbuf);
        nsel++;
      }
    } else {
      /* Eq. 4: bounded heap of the K+1 highest-ranked entries. */
      int64_t cap = K + 1, n = 0;
      for (int64_t j = 0; j < J->Lk; ++j) {
        if (!key_valid(J, bh, i, j)) continue;
        entry e;
        e.j = (int32_t)j;
        e.s = dot_row(J, bh * J->Lk + j, qbuf);
        if (n < cap) {
          heap[n] = e;
          heap_sift_up(heap, (int)n);
          n++;
        } else if (ranks_below(heap[0], e)) {
          heap[0] = e;
          heap_sift_down(heap, (int)n, 0);
        }
      }
      memcpy(sel, heap, sizeof(entry) * (size_t)n);
      qsort(sel, (size_t)n, sizeof(entry), cmp_rank_desc);
      nsel = n > K ? K : n;
      if (n > K) next = sel[K].s;
    }
    if (J->eval_idx || J->vanilla) qsort(sel, (size_t)nsel, sizeof(entry), cmp_rank_desc);

    /* activation over the kept entries only (Eq. 4 / Eq. 3) */
    if (J->act == ACT_SOFTMAX) {
      double m = -INFINITY, z = 0.0;
      for (int64_t t = 0; t < nsel; ++t)
        if (sel[t].s > m) m = sel[t].s;
      for (int64_t t = 0; t < nsel; ++t) {
        w[t] = exp(sel[t].s - m);
        z += w[t];
      }
      for (int64_t t = 0; t < nsel; ++t) w[t] /= z;
    } else {
      for (int64_t t = 0; t < nsel; ++t) w[t] = sel[t].s > 0.0 ? sel[t].s : 0.0;
    }

    /* weighted sum of the kept value rows */
    double* o = J->out ? J->out + r * d : NULL;
    if (o) {
      for (int64_t c = 0; c < d; ++c) o[c] = 0.0;
      for (int64_t t = 0; t < nsel; ++t) {
        const int64_t vrow = bh * J->Lk + sel[t].j;
        for (int64_t c = 0; c < d; ++c) o[c] += w[t] * widen(J->v, (size_t)(vrow * d + c), J->dtype);
      }
    }
    if (J->idx && !J->vanilla) {
      for (int64_t t = 0; t < K; ++t) J->idx[r * K + t] = t < nsel ? sel[t].j : -1;
    }
    if (J->score && !J->vanilla) {
      for (int64_t t = 0; t < K; ++t) J->score[r * K + t] = t < nsel ? sel[t].s : -INFINITY;
    }
    if (J->next_score) J->next_score[r] = next;
  }
done:
  free(qbuf);
  free(heap);
  free(sel);
  free(w);
  return NULL;
}

static int run(job proto, int nthreads) {
  if (proto.d <= 0 || proto.Lq <= 0 || proto.Lk <= 0 || proto.topk < 1) return -2;
  if (nthreads <= 0) nthreads = (int)sysconf(_SC_NPROCESSORS_ONLN);
  if (nthreads < 1) nthreads = 1;
  if (nthreads > proto.nrows) nthreads = (int)(proto.nrows > 0 ? proto.nrows : 1);
  job* jobs = (job*)calloc((size_t)nthreads, sizeof(job));
  pthread_t* th = (pthread_t*)calloc((size_t)nthreads, sizeof(pthread_t));
  if (!jobs || !th) {
    free(jobs);
    free(th);
    return -1;
  }
  int64_t per = (proto.nrows + nthreads - 1) / nthreads;
  for (int t = 0; t < nthreads; ++t) {
    jobs[t] = proto;
    jobs[t].begin = (int64_t)t * per;
    jobs[t].end = jobs[t].begin + per < proto.nrows ? jobs[t].begin + per : proto.nrows;
    if (jobs[t].begin > jobs[t].end) jobs[t].begin = jobs[t].end;
    jobs[t].status = 0;
    pthread_create(&th[t], NULL, run_rows, &jobs[t]);
  }
  int status = 0;
  for (int t = 0; t < nthreads; ++t) {
    pthread_join(th[t], NULL);
    if (jobs[t].status) status = jobs[t].status;
  }
  free(jobs);
  free(th);
  return status;
}

/* Mask arguments shared by the entry points (Eq. 2): causal (requires
 * Lq <= Lk; key j is valid for query i iff j <= i + Lk - Lq), kv_len
 * ([B] int32 or NULL; key j valid iff j < kv_len[b]) and mask (uint32 bit
 * words or NULL; bit j % 32 of word b*mbs + h*mhs + i*ceil(Lk/32) + j/32;
 * 1 = valid).  All three apply together. */
static int set_masks(job* J, int64_t Lq, int64_t Lk, int causal, const int32_t* kv_len, const uint32_t* mask,
                     int64_t mbs, int64_t mhs) {
  if (causal && Lq > Lk) return -2;
  J->causal = causal;
  J->coff = Lk - Lq;
  J->kv_len = kv_len;
  J->mask = mask;
  J->mbs = mbs;
  J->mhs = mhs;
  J->mw = (Lk + 31) / 32;
  return 0;
}

/* Top-k attention (Eq. 4) or, with act = ACT_RELU and B = H = 1, the
 * top-k feed-forward layer (Eq. 3), under the masks above.  Rows are
 * flattened (b, h, i) indices into [B*H*Lq]; rows == NULL means all of them
 * in order.  Outputs per listed row: out [d], idx [topk] (-1 padded), score
 * [topk] (-inf padded), next_score = the (k+1)-th score or -inf. */
int oracle_topk_masked(int act, int dtype, const void* q, const void* k, const void* v, int64_t B, int64_t H,
                       int64_t Lq, int64_t Lk, int64_t d, int64_t topk, int causal, const int32_t* kv_len,
                       const uint32_t* mask, int64_t mbs, int64_t mhs, const int64_t* rows, int64_t nrows,
                       double* out, int32_t* idx, double* score, double* next_score, int nthreads) {
  job J;
  memset(&J, 0, sizeof J);
  J.act = act;
  J.dtype = dtype;
  J.q = q;
  J.k = k;
  J.v = v;
  J.H = H;
  J.Lq = Lq;
  J.Lk = Lk;
  J.d = d;
  J.topk = topk;
  J.rows = rows;
  J.nrows = rows ? nrows : B * H * Lq;
  J.out = out;
  J.idx = idx;
  J.score = score;
  J.next_score = next_score;
  if (set_masks(&J, Lq, Lk, causal, kv_len, mask, mbs, mhs)) return -2;
  return run(J, nthreads);
}

int oracle_topk(int act, int dtype, const void* q, const void* k, const void* v, int64_t B, int64_t H,
                int64_t Lq, int64_t Lk, int64_t d, int64_t topk, int causal, const int64_t* rows,
                int64_t nrows, double* out, int32_t* idx, double* score, double* next_score,
                int nthreads) {
  return oracle_topk_masked(act, dtype, q, k, v, B, H, Lq, Lk, d, topk, causal, NULL, NULL, 0, 0, rows, nrows,
                            out, idx, score, next_score, nthreads);
}

/* Plain attention over every valid key (Eq. 1 under the masks of Eq. 2).
 * Same row convention as oracle_topk. */
int oracle_vanilla_masked(int act, int dtype, const void* q, const void* k, const void* v, int64_t B,
                          int64_t H, int64_t Lq, int64_t Lk, int64_t d, int causal, const int32_t* kv_len,
                          const uint32_t* mask, int64_t mbs, int64_t mhs, const int64_t* rows, int64_t nrows,
                          double* out, int nthreads) {
  job J;
  memset(&J, 0, sizeof J);
  J.act = act;
  J.dtype = dtype;
  J.q = q;
  J.k = k;
  J.v = v;
  J.H = H;
  J.Lq = Lq;
  J.Lk = Lk;
  J.d = d;
  J.topk = Lk;
  J.vanilla = 1;
  J.rows = rows;
  J.nrows = rows ? nrows : B * H * Lq;
  J.out = out;
  if (set_masks(&J, Lq, Lk, causal, kv_len, mask, mbs, mhs)) return -2;
  return run(J, nthreads);
}

int oracle_vanilla(int act, int dtype, const void* q, const void* k, const void* v, int64_t B, int64_t H,
                   int64_t Lq, int64_t Lk, int64_t d, int causal, const int64_t* rows, int64_t nrows,
                   double* out, int nthreads) {
  return oracle_vanilla_masked(act, dtype, q, k, v, B, H, Lq, Lk, d, causal, NULL, NULL, 0, 0, rows, nrows, out,
                               nthreads);
}

/* Index-evaluate: the kept set of each listed row is given in idx
 * ([nrows][topk], -1 = empty slot); scores are recomputed in double and
 * the activation and weighted sum follow Eq. 4 / Eq. 3 from there.  score
 * and, if idx_out is not NULL, idx_out receive the kept entries in the
 * total order (score descending, index ascending), padded with -inf / -1. */
int oracle_eval_indices(int act, int dtype, const void* q, const void* k, const void* v, int64_t B,
                        int64_t H, int64_t Lq, int64_t Lk, int64_t d, int64_t topk,
                        const int64_t* rows, int64_t nrows, const int32_t* idx, double* out,
                        double* score, int32_t* idx_out, int nthreads) {
  job J;
  memset(&J, 0, sizeof J);
  J.act = act;
  J.dtype = dtype;
  J.q = q;
  J.k = k;
  J.v = v;
  J.H = H;
  J.Lq = Lq;
  J.Lk = Lk;
  J.d = d;
  J.topk = topk;
  J.rows = rows;
  J.nrows = rows ? nrows : B * H * Lq;
  J.eval_idx = idx;
  J.out = out;
  J.score = score;
  J.idx = idx_out;
  return run(J, nthreads);
}

/* ------------------------------------------------------------------------
 * Backward pass for a given kept set (Sec. 2.2, "Improving efficiency
 * through top-k attention").  The kept set of every row is the cache the
 * forward pass leaves behind; the selection is piecewise constant in the
 * scores, so the gradient reaches Q and K only through the kept scores.
 * With L = sum_i dout_i . out_i, per row i (problem b, h) with kept keys
 * j_1 .. j_n (idx entries < 0 are empty):
 *
 *   s_t   = q_i . k_{j_t}                    recomputed in double
 *   a_t   = act(s)_t                          softmax over the kept entries
 *                                             (Eq. 4) or ReLU (Eq. 3)
 *   da_t  = dout_i . v_{j_t}                  dL/da_t
 *   ds_t  = a_t (da_t - sum_u a_u da_u)       softmax
 *         = da_t if s_t > 0, else 0           ReLU (derivative 0 at s = 0)
 *   dq_i  = sum_t ds_t k_{j_t}
 *   dk_j  = sum over (i, t) with j_t = j of ds_t q_i
 *   dv_j  = sum over (i, t) with j_t = j of a_t dout_i
 *
 * Phase 1 runs the per-row steps (threads split the rows) and keeps a_t and
 * ds_t; phase 2 forms dk and dv as the two sparse-by-dense products (threads
 * split the keys of each problem into ranges; each key's terms are added in
 * ascending (i, t) order).
 * ---------------------------------------------------------------------- */
typedef struct {
  int act, dtype, dout_dtype;
  const void *q, *k, *v, *dout;
  int64_t Lq, Lk, d, topk;
  const int32_t* idx;
  double *a, *ds, *dq, *dk, *dv;
  int64_t nchunk;     /* key ranges per problem (phase 2) */
  int64_t begin, end; /* rows (phase 1) or (problem, key range) units (phase 2) */
  int status;
} bwd_job;

static void* bwd_rows(void* arg) {
  bwd_job* J = (bwd_job*)arg;
  const int64_t d = J->d, K = J->topk;
  double* qbuf = (double*)malloc(sizeof(double) * (size_t)d);
  double* gbuf = (double*)malloc(sizeof(double) * (size_t)d);
  double* s = (double*)malloc(sizeof(double) * (size_t)K);
  double* da = (double*)malloc(sizeof(double) * (size_t)K);
  if (!qbuf || !gbuf || !s || !da) {
    J->status = -1;
    goto done;
  }
  for (int64_t row = J->begin; row < J->end; ++row) {
    const int64_t bh = row / J->Lq;
    const int32_t* kept = J->idx + row * K;
    double* a = J->a + row * K;
    double* ds = J->ds + row * K;
    for (int64_t c = 0; c < d; ++c) {
      qbuf[c] = widen(J->q, (size_t)(row * d + c), J->dtype);
      gbuf[c] = widen(J->dout, (size_t)(row * d + c), J->dout_dtype);
    }
    /* scores of the kept entries, and dL/da_t */
    for (int64_t t = 0; t < K; ++t) {
      s[t] = 0.0;
      da[t] = 0.0;
      a[t] = 0.0;
      ds[t] = 0.0;
      const int32_t j = kept[t];
      if (j < 0) continue;
      if (j >= J->Lk) {
        J->status = -3;
        continue;
      }
      const int64_t krow = bh * J->Lk + j;
      for (int64_t c = 0; c < d; ++c) {
        s[t] += qbuf[c] * widen(J->k, (size_t)(krow * d + c), J->dtype);
        da[t] += gbuf[c] * widen(J->v, (size_t)(krow * d + c), J->dtype);
      }
    }
    /* activation over the kept entries, then its backward */
    if (J->act == ACT_SOFTMAX) {
      double m = -INFINITY, z = 0.0, dot = 0.0;
      for (int64_t t = 0; t < K; ++t)
        if (kept[t] >= 0 && kept[t] < J->Lk && s[t] > m) m = s[t];
      for (int64_t t = 0; t < K; ++t)
        if (kept[t] >= 0 && kept[t] < J->Lk) {
          a[t] = exp(s[t] - m);
          z += a[t];
        }
      for (int64_t t = 0; t < K; ++t)
        if (kept[t] >= 0 && kept[t] < J->Lk) {
          a[t] /= z;
          dot += a[t] * da[t];
        }
      for (int64_t t = 0; t < K; ++t)
        if (kept[t] >= 0 && kept[t] < J->Lk) ds[t] = a[t] * (da[t] - dot);
    } else {
      for (int64_t t = 0; t < K; ++t)
        if (kept[t] >= 0 && kept[t] < J->Lk) {
          a[t] = s[t] > 0.0 ? s[t] : 0.0;
          ds[t] = s[t] > 0.0 ? da[t] : 0.0;
        }
    }
    /* dq_i = sum_t ds_t k_{j_t} */
    double* dq = J->dq + row * d;
    for (int64_t c = 0; c < d; ++c) dq[c] = 0.0;
    for (int64_t t = 0; t < K; ++t) {
      const int32_t j = kept[t];
      if (j < 0 || j >= J->Lk) continue;
      const int64_t krow = bh * J->Lk + j;
      for (int64_t c = 0; c < d; ++c) dq[c] += ds[t] * widen(J->k, (size_t)(krow * d + c), J->dtype);
    }
  }
done:
  free(qbuf);
  free(gbuf);
  free(s);
  free(da);
  return NULL;
}

/* Phase 2: the units [begin, end) are (problem, key range) pairs, nchunk
 * ranges per problem.  A unit scans its problem's kept sets in ascending
 * (i, t) order and adds each term whose key falls in its range. */
static void* bwd_keys(void* arg) {
  bwd_job* J = (bwd_job*)arg;
  const int64_t d = J->d, K = J->topk, C = J->nchunk;
  for (int64_t u = J->begin; u < J->end; ++u) {
    const int64_t bh = u / C, c = u % C;
    const int64_t j0 = c * J->Lk / C, j1 = (c + 1) * J->Lk / C;
    for (int64_t j = j0; j < j1; ++j)
      for (int64_t e = 0; e < d; ++e) {
        J->dk[(bh * J->Lk + j) * d + e] = 0.0;
        J->dv[(bh * J->Lk + j) * d + e] = 0.0;
      }
    for (int64_t i = 0; i < J->Lq; ++i) {
      const int64_t row = bh * J->Lq + i;
      const int32_t* kept = J->idx + row * K;
      for (int64_t t = 0; t < K; ++t) {
        const int64_t j = kept[t];
        if (j < j0 || j >= j1) continue;
        const double a = J->a[row * K + t], g = J->ds[row * K + t];
        double* dk = J->dk + (bh * J->Lk + j) * d;
        double* dv = J->dv + (bh * J->Lk + j) * d;
        for (int64_t e = 0; e < d; ++e) {
          dk[e] += g * widen(J->q, (size_t)(row * d + e), J->dtype);
          dv[e] += a * widen(J->dout, (size_t)(row * d + e), J->dout_dtype);
        }
      }
    }
  }
  return NULL;
}

static int bwd_run(bwd_job proto, int64_t total, int phase, int nthreads) {
  if (nthreads <= 0) nthreads = (int)sysconf(_SC_NPROCESSORS_ONLN);
  if (nthreads < 1) nthreads = 1;
  if (nthreads > total) nthreads = (int)(total > 0 ? total : 1);
  bwd_job* jobs = (bwd_job*)calloc((size_t)nthreads, sizeof(bwd_job));
  pthread_t* th = (pthread_t*)calloc((size_t)nthreads, sizeof(pthread_t));
  if (!jobs || !th) {
    free(jobs);
    free(th);
    return -1;
  }
  const int64_t per = (total + nthreads - 1) / nthreads;
  for (int t = 0; t < nthreads; ++t) {
    jobs[t] = proto;
    jobs[t].begin = (int64_t)t * per < total ? (int64_t)t * per : total;
    jobs[t].end = jobs[t].begin + per < total ? jobs[t].begin + per : total;
    jobs[t].status = 0;
    pthread_create(&th[t], NULL, phase == 1 ? bwd_rows : bwd_keys, &jobs[t]);
  }
  int status = 0;
  for (int t = 0; t < nthreads; ++t) {
    pthread_join(th[t], NULL);
    if (jobs[t].status) status = jobs[t].status;
  }
  free(jobs);
  free(th);
  return status;
}

/* Gradients of Eq. 4 (act = ACT_SOFTMAX) or Eq. 3 (act = ACT_RELU, with
 * B = H = 1: q = x, k = W1, v = W2) with respect to q, k and v, for the
 * kept sets idx [B*H*Lq][topk] (-1 = empty slot) and the output gradient
 * dout [B*H*Lq][d] (its own dtype code).  Outputs, all rows: dq
 * [B*H*Lq][d], dk and dv [B*H*Lk][d].  Every kept index must be < Lk
 * (-3 otherwise). */
int oracle_topk_bwd(int act, int dtype, const void* q, const void* k, const void* v, int dout_dtype,
                    const void* dout, int64_t B, int64_t H, int64_t Lq, int64_t Lk, int64_t d,
                    int64_t topk, const int32_t* idx, double* dq, double* dk, double* dv, int nthreads) {
  if (d <= 0 || Lq <= 0 || Lk <= 0 || topk < 1 || B <= 0 || H <= 0) return -2;
  bwd_job J;
  memset(&J, 0, sizeof J);
  J.act = act;
  J.dtype = dtype;
  J.dout_dtype = dout_dtype;
  J.q = q;
  J.k = k;
  J.v = v;
  J.dout = dout;
  J.Lq = Lq;
  J.Lk = Lk;
  J.d = d;
  J.topk = topk;
  J.idx = idx;
  J.dq = dq;
  J.dk = dk;
  J.dv = dv;
  const int64_t rows = B * H * Lq;
  J.a = (double*)malloc(sizeof(double) * (size_t)(rows * topk));
  J.ds = (double*)malloc(sizeof(double) * (size_t)(rows * topk));
  int rc = -1;
  if (J.a && J.ds) {
    int nt = nthreads > 0 ? nthreads : (int)sysconf(_SC_NPROCESSORS_ONLN);
    if (nt < 1) nt = 1;
    J.nchunk = nt < Lk ? nt : Lk;
    rc = bwd_run(J, rows, 1, nt);
    if (rc == 0) rc = bwd_run(J, B * H * J.nchunk, 2, nt);
  }
  free(J.a);
  free(J.ds);
  return rc;
}

int oracle_hardware_threads(void) { return (int)sysconf(_SC_NPROCESSORS_ONLN); }
