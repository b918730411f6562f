/*
 * Dynamic Memory Compression (arXiv 2403.09636): CPU fp64 oracle in plain C.
 *
 * TEST INFRASTRUCTURE ONLY. Used by the tests (parity at sizes where the numpy
 * oracle's per-token loop is slow) and by the bench's timed CPU baseline.
 * Shares no code with the CUDA path.
 *
 * For one (layer, sequence, KV head) it runs Algorithm 1 token by token:
 *   alpha_t = round(sigmoid(k_t[0]))     Eq. (reuse); a tie rounds up, NaN -> 0
 *   omega_t = sigmoid(mean_g q_{t,g}[0]) Eq. (reuse); the group mean is the
 *                                        grouped-query reading (G = 1 for MHA)
 *   k_t[0] <- 0                          Algorithm 1, third step
 *   accumulate (alpha = 1, cache not empty):
 *       z <- z + omega;  K_l <- (K_l z_prev + k_t omega) / z;  V_l likewise
 *   append otherwise: new slot (k_t, v_t), z = omega
 * With window = w > 0 (the window-grouping approximation, Sec. 3.3) the last
 * slot is instead the omega-weighted mean of the last min(segment length, w)
 * tokens of its segment, z their summed omega: the open segment's last w
 * tokens are kept and the slot recomputed from them at every merge.
 * And, for decode tokens, softmax attention of every query of the group over
 * the updated cache, Eq. (attn-softmax), with q[0] removed and scale
 * 1/sqrt(d_h) (masking appendix). Everything is double precision; inputs are
 * float (bf16 and fp32 inputs are exact in float).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  int32_t d;          /* head dim */
  int32_t G;          /* queries sharing this KV head (1 for MHA) */
  int32_t n_prompt;   /* prompt tokens, compressed without attention */
  int32_t n_decode;   /* decode tokens: compressed, then attended */
  const float* pk;    /* [n_prompt][d] */
  const float* pv;    /* [n_prompt][d] */
  const float* pq0;   /* [n_prompt][G]: first component of each query */
  const float* dk;    /* [n_decode][d] */
  const float* dv;    /* [n_decode][d] */
  const float* dq;    /* [n_decode][G][d] */
  int32_t cap;        /* slot capacity of K, V, z below */
  double* K;          /* [cap][d] final slots (may be NULL) */
  double* V;          /* [cap][d] */
  double* z;          /* [cap] */
  double* pK;         /* [cap][d] slots right after the prompt (may be NULL) */
  double* pV;         /* [cap][d] */
  double* pz;         /* [cap] */
  int32_t* len_prompt;  /* slots after the prompt */
  int32_t* len_final;   /* slots after the last decode token */
  int32_t* lens;        /* [n_decode] slots after each decode token (may be NULL) */
  double* out;          /* [n_decode][G][d] attention outputs (may be NULL) */
  int32_t status;       /* 0 ok, 1 capacity exceeded, 2 out of memory */
  int32_t window;       /* 0: Algorithm 1; w > 0: window grouping over w tokens */
} dmc_ref_instance;

/* The open segment's last `window` tokens (k with k[0] cleared, v, omega). */
typedef struct {
  int w, n;  /* window, tokens of the segment so far */
  double* k; /* [w][d] ring: token p of the segment at row p % w */
  double* v;
  double* om;
} seg_ring;

static double sigmoid(double x) { return 1.0 / (1.0 + exp(-x)); }

static int decide(double k0) { return sigmoid(k0) >= 0.5 ? 1 : 0; }

static double importance(const float* q0, int G, int stride) {
  double m = 0.0;
  for (int g = 0; g < G; ++g) m += (double)q0[(size_t)g * stride];
  return sigmoid(m / (double)G);
}

/* Algorithm 1 for one token. Returns 0, or 1 when a new slot would not fit. */
static int update(int d, int cap, double* K, double* V, double* z, int* len,
                  const float* k, const float* v, double omega, seg_ring* ring) {
  int alpha = decide((double)k[0]);
  if (ring) {
    /* window grouping: record the token, the last slot is the mean of the
       segment's last w tokens */
    int open = !(alpha == 1 && *len > 0);
    if (open) {
      if (*len >= cap) return 1;
      ring->n = 0;
      *len += 1;
    }
    int row = ring->n % ring->w;
    ring->k[(size_t)row * d] = 0.0;
    for (int i = 1; i < d; ++i) ring->k[(size_t)row * d + i] = (double)k[i];
    for (int i = 0; i < d; ++i) ring->v[(size_t)row * d + i] = (double)v[i];
    ring->om[row] = omega;
    ring->n += 1;
    int m = ring->n < ring->w ? ring->n : ring->w;
    double* Kl = K + (size_t)(*len - 1) * d;
    double* Vl = V + (size_t)(*len - 1) * d;
    double zs = 0.0;
    for (int i = 0; i < d; ++i) { Kl[i] = 0.0; Vl[i] = 0.0; }
    for (int e = 0; e < m; ++e) {
      int r = (ring->n - 1 - e) % ring->w;
      double om = ring->om[r];
      zs += om;
      for (int i = 0; i < d; ++i) {
        Kl[i] += om * ring->k[(size_t)r * d + i];
        Vl[i] += om * ring->v[(size_t)r * d + i];
      }
    }
    for (int i = 0; i < d; ++i) { Kl[i] /= zs; Vl[i] /= zs; }
    z[*len - 1] = zs;
    return 0;
  }
  if (alpha == 1 && *len > 0) {
    int l = *len - 1;
    double z_prev = z[l];
    double z_t = z_prev + omega;
    double* Kl = K + (size_t)l * d;
    double* Vl = V + (size_t)l * d;
    Kl[0] = (Kl[0] * z_prev + 0.0 * omega) / z_t;
    for (int i = 1; i < d; ++i) Kl[i] = (Kl[i] * z_prev + (double)k[i] * omega) / z_t;
    for (int i = 0; i < d; ++i) Vl[i] = (Vl[i] * z_prev + (double)v[i] * omega) / z_t;
    z[l] = z_t;
  } else {
    if (*len >= cap) return 1;
    double* Kn = K + (size_t)(*len) * d;
    double* Vn = V + (size_t)(*len) * d;
    Kn[0] = 0.0;
    for (int i = 1; i < d; ++i) Kn[i] = (double)k[i];
    for (int i = 0; i < d; ++i) Vn[i] = (double)v[i];
    z[*len] = omega;
    *len += 1;
  }
  return 0;
}

/* Eq. (attn-softmax) of one query over `len` slots; s is scratch of len doubles. */
static void attend(int d, int len, const double* K, const double* V,
                   const float* q, double* s, double* o) {
  double scale = 1.0 / sqrt((double)d);
  double mx = -INFINITY;
  for (int j = 0; j < len; ++j) {
    const double* Kj = K + (size_t)j * d;
    double acc = 0.0;  /* q[0] removed: the sum starts at component 1 */
    for (int i = 1; i < d; ++i) acc += (double)q[i] * Kj[i];
    s[j] = acc * scale;
    if (s[j] > mx) mx = s[j];
  }
  double den = 0.0;
  for (int j = 0; j < len; ++j) { s[j] = exp(s[j] - mx); den += s[j]; }
  for (int i = 0; i < d; ++i) o[i] = 0.0;
  for (int j = 0; j < len; ++j) {
    const double* Vj = V + (size_t)j * d;
    double p = s[j] / den;
    for (int i = 0; i < d; ++i) o[i] += p * Vj[i];
  }
}

int dmc_ref_run(dmc_ref_instance* in) {
  int d = in->d, G = in->G, cap = in->cap;
  double* K = in->K ? in->K : (double*)malloc(sizeof(double) * (size_t)cap * d);
  double* V = in->V ? in->V : (double*)malloc(sizeof(double) * (size_t)cap * d);
  double* z = in->z ? in->z : (double*)malloc(sizeof(double) * (size_t)cap);
  double* s = (double*)malloc(sizeof(double) * (size_t)(cap > 0 ? cap : 1));
  int len = 0;
  seg_ring ring_store, *ring = NULL;
  memset(&ring_store, 0, sizeof(ring_store));
  if (in->window > 0) {
    ring_store.w = in->window;
    ring_store.k = (double*)malloc(sizeof(double) * (size_t)in->window * d);
    ring_store.v = (double*)malloc(sizeof(double) * (size_t)in->window * d);
    ring_store.om = (double*)malloc(sizeof(double) * (size_t)in->window);
    ring = &ring_store;
  }
  in->status = 0;
  if (!K || !V || !z || !s || (ring && (!ring->k || !ring->v || !ring->om))) { in->status = 2; goto done; }
  for (int t = 0; t < in->n_prompt; ++t) {
    double w = importance(in->pq0 + (size_t)t * G, G, 1);
    if (update(d, cap, K, V, z, &len, in->pk + (size_t)t * d, in->pv + (size_t)t * d, w, ring)) {
      in->status = 1; goto done;
    }
  }
  if (in->len_prompt) *in->len_prompt = len;
  if (in->pK) memcpy(in->pK, K, sizeof(double) * (size_t)len * d);
  if (in->pV) memcpy(in->pV, V, sizeof(double) * (size_t)len * d);
  if (in->pz) memcpy(in->pz, z, sizeof(double) * (size_t)len);
  for (int t = 0; t < in->n_decode; ++t) {
    const float* qt = in->dq + (size_t)t * G * d;
    double w = importance(qt, G, d);
    if (update(d, cap, K, V, z, &len, in->dk + (size_t)t * d, in->dv + (size_t)t * d, w, ring)) {
      in->status = 1; goto done;
    }
    if (in->lens) in->lens[t] = len;
    if (in->out)
      for (int g = 0; g < G; ++g)
        attend(d, len, K, V, qt + (size_t)g * d, s, in->out + ((size_t)t * G + g) * d);
  }
done:
  if (in->len_final) *in->len_final = len;
  if (!in->K) free(K);
  if (!in->V) free(V);
  if (!in->z) free(z);
  free(s);
  free(ring_store.k);
  free(ring_store.v);
  free(ring_store.om);
  return in->status;
}

typedef struct {
  dmc_ref_instance* inst;
  int n;
  int stride;
  int first;
} worker_arg;

static void* worker(void* p) {
  worker_arg* a = (worker_arg*)p;
  for (int i = a->first; i < a->n; i += a->stride) dmc_ref_run(&a->inst[i]);
  return NULL;
}

/* Runs n independent instances on `threads` POSIX threads (instance i on
 * thread i mod threads). Returns the number of instances with status != 0. */
int dmc_ref_run_many(dmc_ref_instance* inst, int n, int threads) {
  if (threads < 1) threads = 1;
  if (threads > n) threads = n > 0 ? n : 1;
  pthread_t* tid = (pthread_t*)malloc(sizeof(pthread_t) * (size_t)threads);
  worker_arg* args = (worker_arg*)malloc(sizeof(worker_arg) * (size_t)threads);
  for (int t = 0; t < threads; ++t) {
    args[t].inst = inst; args[t].n = n; args[t].stride = threads; args[t].first = t;
    pthread_create(&tid[t], NULL, worker, &args[t]);
  }
  for (int t = 0; t < threads; ++t) pthread_join(tid[t], NULL);
  free(tid);
  free(args);
  int bad = 0;
  for (int i = 0; i < n; ++i) bad += inst[i].status != 0;
  return bad;
}

int dmc_ref_instance_size(void) { return (int)sizeof(dmc_ref_instance); }
