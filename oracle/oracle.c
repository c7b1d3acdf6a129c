/*
 * oracle.c -- plain fp64 CPU oracle for incremental-prefill attention.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path (the CUDA library and
 * its Python binding) includes, links or calls this file.  Only tests/, the
 * smoke check and the CPU-baseline leg of the benchmark load it.
 *
 * What it computes (paper section III-A):
 *   Eq. (k), (v): the layer's key/value vectors are the given inputs here; the
 *                 synthetic Q/K/V stand in for W_Q h, W_K h, W_V h.
 *   Eq. (causal_attention_1..3): a_n = softmax(q_n K_{1:n}^T / sqrt(d_k)),
 *                 o_n = a_n V_{1:n}, with "1:n" meaning every cached key whose
 *                 absolute position does not exceed the query's position.
 *   Rotary position embedding: the paper names none; the rotate-half pairing
 *                 (element i rotates with element i + d/2 by angle
 *                 pos * base^(-2i/d)) is the reading used throughout.
 *   Grouped-query attention: query head h reads key/value head h / (hq/hkv)
 *                 (contiguous grouping), also a reading; the paper is silent.
 *
 * Everything is fp64, written as the definitions read: per (query, head) the
 * visible scores are gathered, the maximum subtracted, exponentiated, summed,
 * and the values averaged with those weights.  Work items (query, head) are
 * independent and are spread over pthreads; no item is split or reordered.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Rotate-half RoPE of x[n][h][d] at absolute positions pos[n] into y. */
void oracle_rope(const double *x, const int64_t *pos, int64_t n, int32_t h,
                 int32_t d, double base, double *y) {
  int32_t half = d / 2;
  for (int64_t t = 0; t < n; ++t) {
    for (int32_t hh = 0; hh < h; ++hh) {
      const double *xr = x + ((size_t)t * h + hh) * d;
      double *yr = y + ((size_t)t * h + hh) * d;
      for (int32_t i = 0; i < half; ++i) {
        double inv_freq = pow(base, -2.0 * (double)i / (double)d);
        double theta = (double)pos[t] * inv_freq;
        double c = cos(theta), s = sin(theta);
        double a = xr[i], b = xr[i + half];
        yr[i] = a * c - b * s;
        yr[i + half] = b * c + a * s;
      }
    }
  }
}

typedef struct {
  const double *q, *k, *v;
  const int64_t *qpos, *kpos;
  int64_t n, nk;
  int32_t hq, hkv, d;
  double scale;
  double *out, *lse;
  int64_t item_begin, item_end; /* items are (t, h) flattened as t*hq + h */
  int status;
} attn_job;

static void *attn_worker(void *arg) {
  attn_job *j = (attn_job *)arg;
  int32_t group = j->hq / j->hkv;
  double *scores = (double *)malloc(sizeof(double) * (size_t)(j->nk > 0 ? j->nk : 1));
  int64_t *idx = (int64_t *)malloc(sizeof(int64_t) * (size_t)(j->nk > 0 ? j->nk : 1));
  if (!scores || !idx) {
    free(scores);
    free(idx);
    j->status = -1;
    return NULL;
  }
  for (int64_t it = j->item_begin; it < j->item_end; ++it) {
    int64_t t = it / j->hq;
    int32_t h = (int32_t)(it % j->hq);
    int32_t kvh = h / group;
    const double *qv = j->q + ((size_t)t * j->hq + h) * j->d;
    double *o = j->out + ((size_t)t * j->hq + h) * j->d;
    /* scores of the visible keys: kpos <= qpos (causal, Eq. causal_attention_1) */
    int64_t m_count = 0;
    for (int64_t tau = 0; tau < j->nk; ++tau) {
      if (j->kpos[tau] > j->qpos[t]) continue;
      const double *kv = j->k + ((size_t)tau * j->hkv + kvh) * j->d;
      double dot = 0.0;
      for (int32_t e = 0; e < j->d; ++e) dot += qv[e] * kv[e];
      scores[m_count] = dot * j->scale;
      idx[m_count] = tau;
      ++m_count;
    }
    for (int32_t e = 0; e < j->d; ++e) o[e] = 0.0;
    if (m_count == 0) {
      if (j->lse) j->lse[(size_t)h * j->n + t] = -INFINITY;
      continue;
    }
    double mx = scores[0];
    for (int64_t a = 1; a < m_count; ++a)
      if (scores[a] > mx) mx = scores[a];
    double z = 0.0;
    for (int64_t a = 0; a < m_count; ++a) {
      scores[a] = exp(scores[a] - mx);
      z += scores[a];
    }
    /* Eq. causal_attention_3: o = sum_tau a_tau v_tau with a = weights / z */
    for (int64_t a = 0; a < m_count; ++a) {
      double w = scores[a] / z;
      const double *vv = j->v + ((size_t)idx[a] * j->hkv + kvh) * j->d;
      for (int32_t e = 0; e < j->d; ++e) o[e] += w * vv[e];
    }
    if (j->lse) j->lse[(size_t)h * j->n + t] = mx + log(z);
  }
  free(scores);
  free(idx);
  j->status = 0;
  return NULL;
}

/*
 * Causal softmax attention with explicit positions.
 *   q[n][hq][d]       (already rotated), qpos[n]
 *   k[nk][hkv][d]     (already rotated), v[nk][hkv][d], kpos[nk]
 *   out[n][hq][d], lse[hq][n] (natural log of the softmax normaliser, may be NULL)
 * Returns 0 on success, -1 on bad arguments or allocation failure.
 */
int oracle_attention(const double *q, const int64_t *qpos, int64_t n,
                     const double *k, const double *v, const int64_t *kpos,
                     int64_t nk, int32_t hq, int32_t hkv, int32_t d,
                     double scale, double *out, double *lse, int32_t threads) {
  if (n < 0 || nk < 0 || hq <= 0 || hkv <= 0 || d <= 0 || hq % hkv != 0)
    return -1;
  if (threads < 1) threads = 1;
  int64_t items = n * (int64_t)hq;
  if (items == 0) return 0;
  if (threads > items) threads = (int32_t)items;
  attn_job *jobs = (attn_job *)calloc((size_t)threads, sizeof(attn_job));
  pthread_t *tids = (pthread_t *)calloc((size_t)threads, sizeof(pthread_t));
  if (!jobs || !tids) {
    free(jobs);
    free(tids);
    return -1;
  }
  for (int32_t w = 0; w < threads; ++w) {
    attn_job *j = &jobs[w];
    j->q = q; j->k = k; j->v = v; j->qpos = qpos; j->kpos = kpos;
    j->n = n; j->nk = nk; j->hq = hq; j->hkv = hkv; j->d = d;
    j->scale = scale; j->out = out; j->lse = lse;
    j->item_begin = items * w / threads;
    j->item_end = items * (w + 1) / threads;
    j->status = -2;
  }
  int32_t started = 0;
  for (int32_t w = 1; w < threads; ++w) {
    if (pthread_create(&tids[w], NULL, attn_worker, &jobs[w]) != 0) break;
    ++started;
  }
  attn_worker(&jobs[0]);
  for (int32_t w = 1; w <= started; ++w) pthread_join(tids[w], NULL);
  /* items of threads that failed to start are computed here, serially */
  for (int32_t w = started + 1; w < threads; ++w) attn_worker(&jobs[w]);
  int rc = 0;
  for (int32_t w = 0; w < threads; ++w)
    if (jobs[w].status != 0) rc = -1;
  free(jobs);
  free(tids);
  return rc;
}
