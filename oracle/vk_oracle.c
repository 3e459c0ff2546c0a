/*
 * vk_oracle.c -- plain, slow, fp64 CPU restatement of the VestigeKV decode hot path.
 *
 * TEST INFRASTRUCTURE ONLY. The test suite, the smoke check and the benchmark's CPU-baseline leg are the
 * only code that may load this library. The CUDA library never calls it, and the two share no code,
 * headers, tables or helpers.
 *
 * Source: "VestigeKV: The NoPE-MLA KV Cache Carries Its Own Sparse-Attention Signal in a Vestigial
 * Branch" (arXiv 2609.03949). Every stored input (bf16 or fp32) is decoded exactly to double and all
 * arithmetic is double. Nothing is blocked, fused or reordered beyond what each definition states.
 *
 * Pinned by tests/test_oracle_pins.py (closed forms, hand cases with a known answer, library routines on
 * special cases, brute force on tiny inputs, the paper's lemmas as invariants). No function here is
 * "parity unpinned".
 *
 * Readings of the paper used here (each listed with its reason in the design notes):
 *   - the cache holds rows 0..N-1; the query sits at position N; the recent window is [N-W, N);
 *   - the archive is A = [n_sink, N-W); k = min(ceil(rho*N), |A|) rows are kept from it per head;
 *   - ties in the top-k go to the smaller position;
 *   - the trigger is row level: Eq. 4, with the content summand either bounded whole by Cauchy-Schwarz
 *     (sketch rank 0, eta_u = |L_u|) or split into a rank-r_sk sketch term and a residual bound, plus a
 *     page-level bound on the RoPE dims that the width-r digest does not cover (reading A); reading B
 *     admits whole 64-row pages by a page-level bound on both summands (sketch rank 0 only).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define D_LAT 512
#define D_ROPE 64
#define PAGE 64

/* Deliberate mistakes for the "known-bad input first" checks: a test sets one, shows that a pin fails,
 * and clears it. 0 = the oracle as written. */
enum {
  MUT_NONE = 0,
  MUT_TIE_LARGER = 1,     /* ties go to the larger position */
  MUT_DROP_WINDOW = 2,    /* the recent window is not attended */
  MUT_SCALE_SQUARED = 3,  /* logits use lambda^2 */
  MUT_ROT_TRANSPOSE = 4,  /* the digest rotation is applied as O^T */
  MUT_DROP_ROPE = 5,      /* attention logits drop the RoPE summand */
  MUT_TRIGGER_NO_Z = 6,   /* trigger ignores the certificate term */
  MUT_SIGMA_ONE_SIDED = 7, /* sigma's inverse DFT drops the factor 2 of the bins that stand for a conjugate pair */
  MUT_PCA_ASCENDING = 8,   /* the PCA basis is ordered by increasing eigenvalue */
  MUT_CONFORMAL_FLOOR = 9, /* the conformal order statistic takes floor((n+1) tau_s) instead of the ceiling */
  MUT_SKETCH_QNORM = 10,   /* with a content sketch, the certificate keeps |qc_h| instead of the residual norm */
};
static int g_mutation = MUT_NONE;
void vko_set_mutation(int m) { g_mutation = m; }

typedef struct {
  int32_t B, H, N;
  int32_t dtype;                              /* 0 = bf16 storage, 1 = fp32 storage */
  const void* latent; int64_t latent_ld, latent_bstride;   /* elements */
  const void* rope;   int64_t rope_ld, rope_bstride;       /* elements */
  const void* q_latent;                       /* [B,H,512] contiguous */
  const void* q_rope;                         /* [B,H,64] contiguous */
} vko_view;

/* ---------------------------------------------------------------- exact decoding of the stored values */
static double from_bf16(uint16_t h) {
  uint32_t bits = (uint32_t)h << 16;
  float f;
  memcpy(&f, &bits, 4);
  return (double)f;
}
static double load(const void* base, int dtype, int64_t i) {
  if (dtype == 1) return (double)((const float*)base)[i];
  return from_bf16(((const uint16_t*)base)[i]);
}
static double L(const vko_view* v, int b, int64_t u, int j) {
  return load(v->latent, v->dtype, (int64_t)b * v->latent_bstride + u * v->latent_ld + j);
}
static double K(const vko_view* v, int b, int64_t u, int j) {
  return load(v->rope, v->dtype, (int64_t)b * v->rope_bstride + u * v->rope_ld + j);
}
static double QC(const vko_view* v, int b, int h, int j) {
  return load(v->q_latent, v->dtype, ((int64_t)b * v->H + h) * D_LAT + j);
}
static double QR(const vko_view* v, int b, int h, int j) {
  return load(v->q_rope, v->dtype, ((int64_t)b * v->H + h) * D_ROPE + j);
}

/* bf16 round-to-nearest-even of a double, straight from the double (no detour through float). */
uint16_t vko_bf16_rne(double x) {
  if (x == 0.0 || !isfinite(x)) {
    float f = (float)x;
    uint32_t b;
    memcpy(&b, &f, 4);
    return (uint16_t)(b >> 16);
  }
  int e;
  double m = frexp(x, &e);              /* x = m * 2^e, 0.5 <= |m| < 1 */
  double scaled = ldexp(m, 8);          /* 8 significant bits -> an integer in [128, 256) */
  double fl = floor(scaled), diff = scaled - fl, q;
  if (diff > 0.5) q = fl + 1.0;
  else if (diff < 0.5) q = fl;
  else q = (fmod(fl, 2.0) == 0.0) ? fl : fl + 1.0;
  float f = (float)ldexp(q, e - 8);     /* exact: 8 significant bits fit a float */
  uint32_t b;
  memcpy(&b, &f, 4);
  return (uint16_t)(b >> 16);
}

/* ---------------------------------------------------------------- set sizes (Sec. 4.1, keep ratio rho) */
/* Archive A = [n_sink, N-W); keep k = min(ceil(rho*N), |A|) archived rows per head. */
int64_t vko_keep_count(int32_t N, double rho, int32_t W, int32_t n_sink) {
  int64_t A = (int64_t)N - W - n_sink;
  if (A < 0) A = 0;
  int64_t k = (int64_t)ceil(rho * (double)N);
  return k < A ? k : A;
}

/* ---------------------------------------------------------------- rotated query (digest scoring) */
/* qt = O * qr (row-major O; the digest keeps its first r coordinates). */
static void rotate64(const float* rot, const double* x, double* y) {
  for (int j = 0; j < D_ROPE; ++j) {
    double acc = 0.0;
    for (int i = 0; i < D_ROPE; ++i) {
      double o = (g_mutation == MUT_ROT_TRANSPOSE) ? (double)rot[i * D_ROPE + j] : (double)rot[j * D_ROPE + i];
      acc += o * x[i];
    }
    y[j] = acc;
  }
}

/* ---------------------------------------------------------------- index build (Sec. 4.2 index entry) */
/* For every row: digest = (O K_u)[0:r] (before rounding; r < 64 only), its bf16 RNE rounding,
 * eta_u = |L_u|_2 (the certificate's row norm with sketch rank 0), and per 64-row page the largest
 * norm of the uncovered RoPE coordinates (O K_u)[r:64] (0 when r = 64). */
void vko_build_index(const vko_view* v, int32_t r, const float* rot, double* digest, uint16_t* digest_bf16,
                     double* eta, double* page_res) {
  const int64_t N = v->N, P = (N + PAGE - 1) / PAGE;
#pragma omp parallel for schedule(static)
  for (int b = 0; b < v->B; ++b) {
    for (int64_t p = 0; p < P; ++p) page_res[(int64_t)b * P + p] = 0.0;
    for (int64_t u = 0; u < N; ++u) {
      double ss = 0.0;
      for (int j = 0; j < D_LAT; ++j) ss += L(v, b, u, j) * L(v, b, u, j);
      eta[(int64_t)b * N + u] = sqrt(ss);
      if (r < D_ROPE) {
        double k[D_ROPE], y[D_ROPE];
        for (int j = 0; j < D_ROPE; ++j) k[j] = K(v, b, u, j);
        rotate64(rot, k, y);
        for (int j = 0; j < r; ++j) {
          digest[((int64_t)b * N + u) * r + j] = y[j];
          if (digest_bf16) digest_bf16[((int64_t)b * N + u) * r + j] = vko_bf16_rne(y[j]);
        }
        double res = 0.0;
        for (int j = r; j < D_ROPE; ++j) res += y[j] * y[j];
        res = sqrt(res);
        double* pr = &page_res[(int64_t)b * P + u / PAGE];
        if (res > *pr) *pr = res;
      }
    }
  }
}

/* ---------------------------------------------------------------- scores (Eq. 4, exact summand) */
/* a[b,h,u] = qr_h . K_u over the 64 RoPE columns (r = 64), or, for a width-r digest,
 * a = (O qr_h)[0:r] . digest_u with the stored bf16 digest. The attention scale is applied later. */
void vko_scores(const vko_view* v, int32_t r, const float* rot, const uint16_t* digest, double* a) {
  const int64_t N = v->N;
#pragma omp parallel for collapse(2) schedule(static)
  for (int b = 0; b < v->B; ++b) {
    for (int h = 0; h < v->H; ++h) {
      double q[D_ROPE], qt[D_ROPE];
      for (int j = 0; j < D_ROPE; ++j) q[j] = QR(v, b, h, j);
      if (r < D_ROPE) rotate64(rot, q, qt);
      double* out = &a[((int64_t)b * v->H + h) * N];
      for (int64_t u = 0; u < N; ++u) {
        double acc = 0.0;
        if (r == D_ROPE) {
          for (int j = 0; j < D_ROPE; ++j) acc += q[j] * K(v, b, u, j);
        } else {
          for (int j = 0; j < r; ++j) acc += qt[j] * from_bf16(digest[((int64_t)b * N + u) * r + j]);
        }
        out[u] = acc;
      }
    }
  }
}

/* ---------------------------------------------------------------- selection (Sec. 4.1) */
typedef struct { double key; int32_t u; } item;

static int by_key_desc_pos_asc(const void* x, const void* y) {
  const item* a = (const item*)x;
  const item* b = (const item*)y;
  if (a->key > b->key) return -1;
  if (a->key < b->key) return 1;
  if (g_mutation == MUT_TIE_LARGER) return (a->u > b->u) ? -1 : (a->u < b->u);
  return (a->u < b->u) ? -1 : (a->u > b->u);
}

/* Per (b,h): sort the archive by (score desc, position asc), keep the first k; the attended set is that
 * together with the sinks [0, n_sink) and the recent window [N-W, N), listed in ascending position.
 * kth = the k-th largest archive score (+inf when k = 0). count = k + W + n_sink. */
void vko_select(int32_t B, int32_t H, int32_t N, const double* a, int64_t k, int32_t W, int32_t n_sink,
                int32_t cap, int32_t* idx, int32_t* count, double* kth) {
#pragma omp parallel for collapse(2) schedule(dynamic)
  for (int b = 0; b < B; ++b) {
    for (int h = 0; h < H; ++h) {
      const double* s = &a[((int64_t)b * H + h) * N];
      int64_t lo = n_sink, hi = (int64_t)N - W;
      int64_t na = hi > lo ? hi - lo : 0;
      item* it = (item*)malloc(sizeof(item) * (size_t)(na > 0 ? na : 1));
      for (int64_t i = 0; i < na; ++i) { it[i].key = s[lo + i]; it[i].u = (int32_t)(lo + i); }
      qsort(it, (size_t)na, sizeof(item), by_key_desc_pos_asc);
      char* mark = (char*)calloc((size_t)N + 1, 1);
      for (int64_t i = 0; i < k && i < na; ++i) mark[it[i].u] = 1;
      for (int64_t u = 0; u < n_sink && u < N; ++u) mark[u] = 1;
      if (g_mutation != MUT_DROP_WINDOW)
        for (int64_t u = hi > 0 ? hi : 0; u < N; ++u) mark[u] = 1;
      int32_t c = 0;
      int32_t* out = &idx[((int64_t)b * H + h) * cap];
      for (int64_t u = 0; u < N; ++u)
        if (mark[u]) { if (c < cap) out[c] = (int32_t)u; ++c; }
      count[b * H + h] = c;
      kth[b * H + h] = (k > 0 && na > 0) ? it[(k < na ? k : na) - 1].key : INFINITY;
      free(mark);
      free(it);
    }
  }
}

/* ---------------------------------------------------------------- attention (Eq. 1, Lemma 1) */
/* Absorbed MLA over an attended set: s_u = lambda*(qc_h . L_u + qr_h . K_u); softmax over the set;
 * the output is the 512-wide latent combination sum_u p_u L_u (the value up-projection W_UV is applied
 * outside the cache read). lse = max + log(sum exp(s - max)); smax = the max logit s*.
 * An empty set gives out = 0, lse = smax = -inf. */
static double logit(const vko_view* v, int b, int h, int64_t u, double lam) {
  double acc = 0.0;
  for (int j = 0; j < D_LAT; ++j) acc += QC(v, b, h, j) * L(v, b, u, j);
  if (g_mutation != MUT_DROP_ROPE)
    for (int j = 0; j < D_ROPE; ++j) acc += QR(v, b, h, j) * K(v, b, u, j);
  return (g_mutation == MUT_SCALE_SQUARED ? lam * lam : lam) * acc;
}

void vko_attention(const vko_view* v, double lam, const int32_t* idx, const int32_t* count, int32_t cap,
                   double* out, double* lse, double* smax) {
#pragma omp parallel for collapse(2) schedule(dynamic)
  for (int b = 0; b < v->B; ++b) {
    for (int h = 0; h < v->H; ++h) {
      const int32_t* set = &idx[((int64_t)b * v->H + h) * cap];
      int32_t n = count[b * v->H + h];
      if (n > cap) n = cap;
      double* o = &out[((int64_t)b * v->H + h) * D_LAT];
      for (int j = 0; j < D_LAT; ++j) o[j] = 0.0;
      if (n <= 0) { lse[b * v->H + h] = -INFINITY; smax[b * v->H + h] = -INFINITY; continue; }
      double* s = (double*)malloc(sizeof(double) * (size_t)n);
      double m = -INFINITY;
      for (int32_t i = 0; i < n; ++i) { s[i] = logit(v, b, h, set[i], lam); if (s[i] > m) m = s[i]; }
      double z = 0.0;
      for (int32_t i = 0; i < n; ++i) z += exp(s[i] - m);
      for (int32_t i = 0; i < n; ++i) {
        double p = exp(s[i] - m) / z;
        for (int j = 0; j < D_LAT; ++j) o[j] += p * L(v, b, set[i], j);
      }
      lse[b * v->H + h] = m + log(z);
      smax[b * v->H + h] = m;
      free(s);
    }
  }
}

/* ---------------------------------------------------------------- recall trigger (Eq. 4, Lemma 2) */
/* With sketch rank 0 the content summand is bounded by Cauchy-Schwarz: |qc_h . L_u| <= |qc_h| eta_u.
 * For a width-r digest the RoPE dims it leaves out are bounded the same way, page by page:
 * |(O qr_h)[r:] . (O K_u)[r:]| <= |(O qr_h)[r:]| page_res[u/64]. The trigger score of an archived row
 * not already attended is
 *     T = lambda * (a[h,u] + |(O qr_h)[r:]| * page_res[page(u)] + z_eff * |qc_h| * eta_u)
 * and the row fires when T > s*_h, the attended set's max logit. With top_j > 0 only the top_j fired
 * rows by (T desc, position asc) are kept. Fired ids are listed in ascending position.
 * With a rank-r_sk content sketch (r_sk > 0: sk16 the stored bf16 entries [B][N][r_sk], p [B][H][r_sk] and rho [B][H]
 * from vko_sketch_query, eta the sketch residual norms from vko_build_sketch) the content summand is the sketch term
 * plus the residual bound of Lemma 1:
 *     T = lambda * (a[h,u] + |(O qr_h)[r:]| * page_res[page(u)] + p_h . s_u + z_eff * rho_h * eta_u). */
void vko_trigger(const vko_view* v, int32_t r, const float* rot, double lam, double z_eff, int32_t top_j,
                 const double* a, const double* eta, const double* page_res, int32_t r_sk, const uint16_t* sk16,
                 const double* p, const double* rho, const int32_t* idx, const int32_t* count, int32_t cap,
                 const double* smax, int32_t W, int32_t n_sink, int32_t capf, int32_t* fidx, int32_t* fcount) {
  const int64_t N = v->N, P = (N + PAGE - 1) / PAGE;
#pragma omp parallel for collapse(2) schedule(dynamic)
  for (int b = 0; b < v->B; ++b) {
    for (int h = 0; h < v->H; ++h) {
      double q[D_ROPE], qt[D_ROPE], qres = 0.0, qcn = 0.0;
      for (int j = 0; j < D_ROPE; ++j) q[j] = QR(v, b, h, j);
      if (r < D_ROPE) {
        rotate64(rot, q, qt);
        for (int j = r; j < D_ROPE; ++j) qres += qt[j] * qt[j];
        qres = sqrt(qres);
      }
      for (int j = 0; j < D_LAT; ++j) qcn += QC(v, b, h, j) * QC(v, b, h, j);
      qcn = sqrt(qcn);
      double zz = (g_mutation == MUT_TRIGGER_NO_Z) ? 0.0 : z_eff;
      const int64_t bh = (int64_t)b * v->H + h;
      const double cert = (r_sk > 0 && g_mutation != MUT_SKETCH_QNORM) ? rho[bh] : qcn;

      char* in_set = (char*)calloc((size_t)N + 1, 1);
      const int32_t* set = &idx[((int64_t)b * v->H + h) * cap];
      int32_t n = count[b * v->H + h];
      if (n > cap) n = cap;
      for (int32_t i = 0; i < n; ++i) in_set[set[i]] = 1;
      double sstar = smax[b * v->H + h];
      const double* s = &a[((int64_t)b * v->H + h) * N];

      int64_t lo = n_sink, hi = N - W;
      item* fired = (item*)malloc(sizeof(item) * (size_t)(hi > lo ? hi - lo : 1));
      int64_t nf = 0;
      for (int64_t u = lo; u < hi; ++u) {
        if (in_set[u]) continue;
        double skt = 0.0;
        for (int j = 0; j < r_sk; ++j) skt += p[bh * r_sk + j] * from_bf16(sk16[((int64_t)b * N + u) * r_sk + j]);
        double t = lam * (s[u] + qres * page_res[(int64_t)b * P + u / PAGE] + skt + zz * cert * eta[(int64_t)b * N + u]);
        if (t > sstar) { fired[nf].key = t; fired[nf].u = (int32_t)u; ++nf; }
      }
      if (top_j > 0 && nf > top_j) {
        qsort(fired, (size_t)nf, sizeof(item), by_key_desc_pos_asc);
        nf = top_j;
      }
      char* mark = (char*)calloc((size_t)N + 1, 1);
      for (int64_t i = 0; i < nf; ++i) mark[fired[i].u] = 1;
      int32_t c = 0;
      int32_t* out = &fidx[((int64_t)b * v->H + h) * capf];
      for (int64_t u = 0; u < N; ++u)
        if (mark[u]) { if (c < capf) out[c] = (int32_t)u; ++c; }
      fcount[b * v->H + h] = c;
      free(mark);
      free(fired);
      free(in_set);
    }
  }
}

/* ---------------------------------------------------------------- page-level trigger (reading B) */
/* Per 64-row page P: the largest RoPE-key norm max_{u in P} |K_u| (all 64 stored dims) and the largest latent
 * norm max_{u in P} eta_u = max |L_u|. Cauchy-Schwarz on both summands of the logit gives, for every row u of P
 * and any query, s(u) = lambda (qc . L_u + qr . K_u) <= lambda (|qr| max_P |K_u| + |qc| max_P eta_u) (Lemma 2
 * with the sketch rank 0, applied to the page's extreme norms instead of the row's own). */
void vko_page_norms(const vko_view* v, double* page_knorm, double* page_eta) {
  const int64_t N = v->N, P = (N + PAGE - 1) / PAGE;
#pragma omp parallel for schedule(static)
  for (int b = 0; b < v->B; ++b) {
    for (int64_t p = 0; p < P; ++p) { page_knorm[(int64_t)b * P + p] = 0.0; page_eta[(int64_t)b * P + p] = 0.0; }
    for (int64_t u = 0; u < N; ++u) {
      double kk = 0.0, ll = 0.0;
      for (int j = 0; j < D_ROPE; ++j) kk += K(v, b, u, j) * K(v, b, u, j);
      for (int j = 0; j < D_LAT; ++j) ll += L(v, b, u, j) * L(v, b, u, j);
      double* pk = &page_knorm[(int64_t)b * P + u / PAGE];
      double* pe = &page_eta[(int64_t)b * P + u / PAGE];
      if (sqrt(kk) > *pk) *pk = sqrt(kk);
      if (sqrt(ll) > *pe) *pe = sqrt(ll);
    }
  }
}

/* Reading B of the recall trigger: a whole archived page is admitted when its page-level bound
 *     Bp = lambda * (|qr_h| * page_knorm[P] + z_eff * |qc_h| * page_eta[P])
 * beats s*_h; its archived rows outside S_h fire. With z_eff >= 1 this is sound (no row left out can beat s*).
 * With top_j > 0 only the top_j fired rows by (Bp desc, position asc) are kept. Fired ids in ascending position. */
void vko_trigger_page(const vko_view* v, double lam, double z_eff, int32_t top_j, const double* page_knorm,
                      const double* page_eta, const int32_t* idx, const int32_t* count, int32_t cap,
                      const double* smax, int32_t W, int32_t n_sink, int32_t capf, int32_t* fidx, int32_t* fcount) {
  const int64_t N = v->N, P = (N + PAGE - 1) / PAGE;
#pragma omp parallel for collapse(2) schedule(dynamic)
  for (int b = 0; b < v->B; ++b) {
    for (int h = 0; h < v->H; ++h) {
      double qrn = 0.0, qcn = 0.0;
      for (int j = 0; j < D_ROPE; ++j) qrn += QR(v, b, h, j) * QR(v, b, h, j);
      for (int j = 0; j < D_LAT; ++j) qcn += QC(v, b, h, j) * QC(v, b, h, j);
      qrn = sqrt(qrn);
      qcn = sqrt(qcn);
      double zz = (g_mutation == MUT_TRIGGER_NO_Z) ? 0.0 : z_eff;
      char* in_set = (char*)calloc((size_t)N + 1, 1);
      const int32_t* set = &idx[((int64_t)b * v->H + h) * cap];
      int32_t n = count[b * v->H + h];
      if (n > cap) n = cap;
      for (int32_t i = 0; i < n; ++i) in_set[set[i]] = 1;
      const double sstar = smax[b * v->H + h];
      int64_t lo = n_sink, hi = N - W;
      item* fired = (item*)malloc(sizeof(item) * (size_t)(hi > lo ? hi - lo : 1));
      int64_t nf = 0;
      for (int64_t u = lo; u < hi; ++u) {
        if (in_set[u]) continue;
        const int64_t pg = (int64_t)b * P + u / PAGE;
        const double bound = lam * (qrn * page_knorm[pg] + zz * qcn * page_eta[pg]);
        if (bound > sstar) { fired[nf].key = bound; fired[nf].u = (int32_t)u; ++nf; }
      }
      if (top_j > 0 && nf > top_j) {
        qsort(fired, (size_t)nf, sizeof(item), by_key_desc_pos_asc);
        nf = top_j;
      }
      char* mark = (char*)calloc((size_t)N + 1, 1);
      for (int64_t i = 0; i < nf; ++i) mark[fired[i].u] = 1;
      int32_t c = 0;
      int32_t* out = &fidx[((int64_t)b * v->H + h) * capf];
      for (int64_t u = 0; u < N; ++u)
        if (mark[u]) { if (c < capf) out[c] = (int32_t)u; ++c; }
      fcount[b * v->H + h] = c;
      free(mark);
      free(fired);
      free(in_set);
    }
  }
}

/* ---------------------------------------------------------------- one decode step */
/* The content sketch's index and query parts (defined with the sketch, below). */
void vko_build_sketch(const vko_view* v, int32_t r_sk, const double* vb, double* s, uint16_t* s16, double* eta);
void vko_sketch_query(const vko_view* v, int32_t r_sk, const double* vb, double* p, double* rho);

/* Score -> select -> attend; in two-tier mode also index -> trigger -> attend over S u F, which equals
 * the LSE merge of the two partial softmaxes (Lemma 1). trigger: 0 off, 1 the row-level rule (reading A),
 * 2 the page-level rule (reading B). With r_sk > 0 the row-level rule uses the rank-r_sk content sketch of basis
 * vb [r_sk][512]; sketch16 is the stored index entry (NULL: the bf16 rounding of vb L_u). idx lists S_h (ascending)
 * followed by F_h (ascending); count = |S_h| + |F_h|. Returns 0, -1 for a sketch with the page-level rule, or -4
 * when a list does not fit in cap. */
int vko_decode_step(const vko_view* v, double rho, int32_t r, int32_t W, int32_t n_sink, double lam,
                    int32_t trigger, double z_eff, int32_t top_j, const float* rot, const uint16_t* digest,
                    int32_t r_sk, const double* vb, const uint16_t* sketch16, int32_t cap, double* out,
                    double* lse, double* smax, int32_t* idx, int32_t* count, double* kth) {
  const int64_t BH = (int64_t)v->B * v->H, N = v->N, P = (N + PAGE - 1) / PAGE;
  int rc = 0;
  if (r_sk > 0 && trigger == 2) return -1;
  double* a = (double*)malloc(sizeof(double) * (size_t)(BH * N));
  vko_scores(v, r, rot, digest, a);
  int64_t k = vko_keep_count(v->N, rho, W, n_sink);
  vko_select(v->B, v->H, v->N, a, k, W, n_sink, cap, idx, count, kth);
  for (int64_t i = 0; i < BH; ++i) if (count[i] > cap) rc = -4;
  vko_attention(v, lam, idx, count, cap, out, lse, smax);
  if (trigger) {
    double* eta = (double*)malloc(sizeof(double) * (size_t)(v->B * N));
    double* pres = (double*)malloc(sizeof(double) * (size_t)(v->B * P));
    double* dig = (r < D_ROPE) ? (double*)malloc(sizeof(double) * (size_t)(v->B * N * r)) : NULL;
    vko_build_index(v, r, rot, dig, NULL, eta, pres);
    int32_t capf = (int32_t)N;
    int32_t* fidx = (int32_t*)malloc(sizeof(int32_t) * (size_t)(BH * capf));
    int32_t* fcount = (int32_t*)malloc(sizeof(int32_t) * (size_t)BH);
    if (trigger == 2) {
      double* pk = (double*)malloc(sizeof(double) * (size_t)(v->B * P));
      double* pe = (double*)malloc(sizeof(double) * (size_t)(v->B * P));
      vko_page_norms(v, pk, pe);
      vko_trigger_page(v, lam, z_eff, top_j, pk, pe, idx, count, cap, smax, W, n_sink, capf, fidx, fcount);
      free(pk);
      free(pe);
    } else if (r_sk > 0) {
      uint16_t* own16 = NULL;
      if (!sketch16) own16 = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)(v->B * N * r_sk));
      vko_build_sketch(v, r_sk, vb, NULL, own16, eta);
      double* pq = (double*)malloc(sizeof(double) * (size_t)(BH * r_sk));
      double* rq = (double*)malloc(sizeof(double) * (size_t)BH);
      vko_sketch_query(v, r_sk, vb, pq, rq);
      vko_trigger(v, r, rot, lam, z_eff, top_j, a, eta, pres, r_sk, sketch16 ? sketch16 : own16, pq, rq, idx, count,
                  cap, smax, W, n_sink, capf, fidx, fcount);
      free(rq);
      free(pq);
      free(own16);
    } else {
      vko_trigger(v, r, rot, lam, z_eff, top_j, a, eta, pres, 0, NULL, NULL, NULL, idx, count, cap, smax, W, n_sink,
                  capf, fidx, fcount);
    }
    for (int64_t i = 0; i < BH; ++i) {
      int32_t* dst = &idx[i * cap];
      int32_t c = count[i];
      for (int32_t j = 0; j < fcount[i]; ++j, ++c)
        if (c < cap) dst[c] = fidx[i * capf + j];
      if (c > cap) rc = -4;
      count[i] = c;
    }
    double* smax_s = (double*)malloc(sizeof(double) * (size_t)BH);
    vko_attention(v, lam, idx, count, cap, out, lse, smax_s);
    free(smax_s);
    free(fidx); free(fcount); free(eta); free(pres); free(dig);
  }
  free(a);
  return rc;
}

/* ---------------------------------------------------------------- sigma selector (Sec. 4.1, Eq. 3) */
/* The query-independent ranking of the paper's tier 1. The branch vectors r_u (the 64 RoPE-branch columns of each
   row, fp64, [N][64] row-major) are cut into fixed blocks of T rows; only whole blocks [jT, (j+1)T) are closed.
   Within a closed block, for each of the 64 dims, the sequence-axis DFT X_k = sum_u r_u e^{-2 pi i k u / T} is kept
   on bins 0 <= k < kappa (and k <= T/2, the one-sided spectrum of a real signal) and inverted:
     low_u = (1/T) sum_{k kept} w_k (A_k cos(2 pi k u / T) + B_k sin(2 pi k u / T)),
   A_k = sum_u r_u cos(2 pi k u / T), B_k = sum_u r_u sin(2 pi k u / T), w_0 = 1, w_{T/2} = 1 (T even), else w_k = 2
   (bin k stands for itself and its conjugate T - k). sigma_u = || r_u - low_u ||_2 over the 64 dims. The sums are
   written out (no FFT). Rows past the last closed block (the open tail) get sigma = -1. */
void vko_sigma(const double* r, int64_t N, int32_t T, int32_t kappa, double* sigma) {
  const int64_t nb = N / T;
  int32_t nk = kappa < T / 2 + 1 ? kappa : T / 2 + 1;      /* kept bins */
  if (nk < 0) nk = 0;
  const double TWO_PI = 6.283185307179586476925286766559;
  double* cs = (double*)malloc(sizeof(double) * (size_t)nk * (size_t)T);
  double* sn = (double*)malloc(sizeof(double) * (size_t)nk * (size_t)T);
  for (int32_t k = 0; k < nk; ++k)
    for (int32_t u = 0; u < T; ++u) {
      const double ang = TWO_PI * (double)(((int64_t)k * u) % T) / (double)T;   /* reduced exactly before cos/sin */
      cs[(size_t)k * T + u] = cos(ang);
      sn[(size_t)k * T + u] = sin(ang);
    }
  for (int64_t u = nb * (int64_t)T; u < N; ++u) sigma[u] = -1.0;
#pragma omp parallel for schedule(static)
  for (int64_t j = 0; j < nb; ++j) {
    const double* rb = r + (size_t)j * T * D_ROPE;
    double* res2 = (double*)calloc((size_t)T, sizeof(double));   /* squared residual per row */
    double* low = (double*)malloc(sizeof(double) * (size_t)T);
    for (int d = 0; d < D_ROPE; ++d) {
      for (int32_t u = 0; u < T; ++u) low[u] = 0.0;
      for (int32_t k = 0; k < nk; ++k) {
        double A = 0.0, B = 0.0;
        for (int32_t u = 0; u < T; ++u) {
          const double x = rb[(size_t)u * D_ROPE + d];
          A += x * cs[(size_t)k * T + u];
          B += x * sn[(size_t)k * T + u];
        }
        double w = (k == 0 || 2 * k == T) ? 1.0 : 2.0;
        if (g_mutation == MUT_SIGMA_ONE_SIDED) w = 1.0;
        for (int32_t u = 0; u < T; ++u) low[u] += w * (A * cs[(size_t)k * T + u] + B * sn[(size_t)k * T + u]);
      }
      for (int32_t u = 0; u < T; ++u) {
        const double e = rb[(size_t)u * D_ROPE + d] - low[u] / (double)T;
        res2[u] += e * e;
      }
    }
    for (int32_t u = 0; u < T; ++u) sigma[(size_t)j * T + u] = sqrt(res2[u]);
    free(res2);
    free(low);
  }
  free(cs);
  free(sn);
}

/* The attended set of the sigma selector (Sec. 4.1): the sinks [0, n_sink), the open tail (rows past the last
   closed block of T rows), and the m closed rows outside the sinks with the largest sigma (ties: the smaller
   position). m is clamped to the number of such rows. Writes the ascending ids to out (room for N) and returns
   their count. */
static const double* g_sig;
static int cmp_sigma(const void* x, const void* y) {
  const int64_t a = *(const int64_t*)x, b = *(const int64_t*)y;
  if (g_sig[a] > g_sig[b]) return -1;
  if (g_sig[a] < g_sig[b]) return 1;
  return (a > b) - (a < b);
}
int64_t vko_sigma_select(const double* sigma, int64_t N, int32_t T, int32_t n_sink, int64_t m, int32_t* out) {
  const int64_t closed = (N / T) * (int64_t)T;
  const int64_t lo = n_sink < closed ? n_sink : closed;
  int64_t nc = closed - lo;
  if (m > nc) m = nc;
  if (m < 0) m = 0;
  int64_t* ord = (int64_t*)malloc(sizeof(int64_t) * (size_t)(nc > 0 ? nc : 1));
  for (int64_t i = 0; i < nc; ++i) ord[i] = lo + i;
  g_sig = sigma;
  qsort(ord, (size_t)nc, sizeof(int64_t), cmp_sigma);
  unsigned char* keep = (unsigned char*)calloc((size_t)(N > 0 ? N : 1), 1);
  for (int64_t i = 0; i < N; ++i) keep[i] = (i < n_sink || i >= closed) ? 1 : 0;
  for (int64_t i = 0; i < m; ++i) keep[ord[i]] = 1;
  int64_t c = 0;
  for (int64_t i = 0; i < N; ++i)
    if (keep[i]) out[c++] = (int32_t)i;
  free(ord);
  free(keep);
  return c;
}

/* ---------------------------------------------------------------- PCA-truncated digest (appendix ablation) */
/* The branch-width ablation keeps the leading principal directions of the RoPE branch instead of the first
 * coordinates after a random rotation. The basis is the eigenvector set of the (uncentred) second-moment matrix
 * M = sum over every row of every sequence of K_u K_u^T (64 x 64, fp64), by decreasing eigenvalue: the rows of the
 * returned rotation, so that digest = (O K_u)[0:r] keeps the most branch energy. Eigenvectors come from the cyclic
 * Jacobi method (a rotation zeroes each off-diagonal pair in turn, sweeps repeat until the off-diagonal mass is
 * negligible); each is signed so that its entry of largest magnitude is positive. eig receives the eigenvalues. */
void vko_second_moment(const vko_view* v, double* M) {
  for (int i = 0; i < D_ROPE * D_ROPE; ++i) M[i] = 0.0;
  for (int b = 0; b < v->B; ++b)
    for (int64_t u = 0; u < v->N; ++u) {
      double k[D_ROPE];
      for (int j = 0; j < D_ROPE; ++j) k[j] = K(v, b, u, j);
      for (int i = 0; i < D_ROPE; ++i)
        for (int j = 0; j < D_ROPE; ++j) M[i * D_ROPE + j] += k[i] * k[j];
    }
}

/* Eigenvalues (descending; ties: the lower index first) and eigenvectors (rows of vec, each signed so that its entry
 * of largest magnitude is positive) of a symmetric n x n matrix by the cyclic Jacobi method. */
static void jacobi_eig(int n, const double* M_in, double* eig, double* vec) {
  double* A = (double*)malloc(sizeof(double) * (size_t)n * n);
  double* V = (double*)malloc(sizeof(double) * (size_t)n * n);
  for (int i = 0; i < n * n; ++i) A[i] = M_in[i];
  for (int i = 0; i < n; ++i)
    for (int j = 0; j < n; ++j) V[i * n + j] = (i == j) ? 1.0 : 0.0;
  double total = 0.0;
  for (int i = 0; i < n * n; ++i) total += A[i] * A[i];
  for (int sweep = 0; sweep < 100; ++sweep) {
    double off = 0.0;
    for (int i = 0; i < n; ++i)
      for (int j = 0; j < n; ++j)
        if (i != j) off += A[i * n + j] * A[i * n + j];
    if (off <= 1e-30 * total) break;
    for (int p = 0; p < n - 1; ++p)
      for (int q = p + 1; q < n; ++q) {
        const double apq = A[p * n + q];
        if (apq == 0.0) continue;
        /* the rotation in the (p, q) plane that zeroes A[p][q] */
        const double theta = (A[q * n + q] - A[p * n + p]) / (2.0 * apq);
        const double t = (theta >= 0.0 ? 1.0 : -1.0) / (fabs(theta) + sqrt(theta * theta + 1.0));
        const double c = 1.0 / sqrt(t * t + 1.0), sn = t * c;
        for (int k = 0; k < n; ++k) {            /* A <- A J (columns p, q) */
          const double akp = A[k * n + p], akq = A[k * n + q];
          A[k * n + p] = c * akp - sn * akq;
          A[k * n + q] = sn * akp + c * akq;
        }
        for (int k = 0; k < n; ++k) {            /* A <- J^T A (rows p, q) */
          const double apk = A[p * n + k], aqk = A[q * n + k];
          A[p * n + k] = c * apk - sn * aqk;
          A[q * n + k] = sn * apk + c * aqk;
        }
        for (int k = 0; k < n; ++k) {            /* V <- V J: column j of V is eigenvector j */
          const double vkp = V[k * n + p], vkq = V[k * n + q];
          V[k * n + p] = c * vkp - sn * vkq;
          V[k * n + q] = sn * vkp + c * vkq;
        }
      }
  }
  /* order by eigenvalue, descending (ties: the lower index first) */
  int* ord = (int*)malloc(sizeof(int) * (size_t)n);
  for (int i = 0; i < n; ++i) ord[i] = i;
  for (int i = 1; i < n; ++i) {
    const int x = ord[i];
    int j = i - 1;
    const int asc = g_mutation == MUT_PCA_ASCENDING;
    while (j >= 0 && (asc ? A[ord[j] * n + ord[j]] > A[x * n + x] : A[ord[j] * n + ord[j]] < A[x * n + x])) {
      ord[j + 1] = ord[j];
      --j;
    }
    ord[j + 1] = x;
  }
  for (int i = 0; i < n; ++i) {
    const int c = ord[i];
    eig[i] = A[c * n + c];
    int big = 0;
    for (int k = 1; k < n; ++k)
      if (fabs(V[k * n + c]) > fabs(V[big * n + c])) big = k;
    const double sg = V[big * n + c] < 0.0 ? -1.0 : 1.0;
    for (int k = 0; k < n; ++k) vec[i * n + k] = sg * V[k * n + c];
  }
  free(ord);
  free(V);
  free(A);
}

void vko_sym_eig(const double* M_in, double* eig, double* vec /* [64][64], row i = eigenvector i */) {
  jacobi_eig(D_ROPE, M_in, eig, vec);
}

void vko_pca_basis(const vko_view* v, double* eig, double* rot) {
  double M[D_ROPE * D_ROPE];
  vko_second_moment(v, M);
  vko_sym_eig(M, eig, rot);
}

/* ---------------------------------------------------------------- content sketch (Sec. 4.2, Eq. 4, Lemma 1) */
/* A rank-r_sk sketch of the content summand. V_r is r_sk orthonormal directions of the 512-wide content space, stored
 * as the rows of vb [r_sk][512]. Lemma 1 splits the content logit of query q and row L as
 *     q . L = (V_r^T q) . (V_r^T L) + delta,   |delta| <= |(I - V_r V_r^T) q| |(I - V_r V_r^T) L|,
 * so the index keeps per row s_u = V_r^T L_u (stored in bf16) and eta_u = |(I - V_r V_r^T) L_u|, and the trigger
 * takes per query p_h = V_r^T qc_h and rho_h = |(I - V_r V_r^T) qc_h|.
 *
 * The basis comes from the context's own queries: the r_sk leading eigenvectors of their uncentred second moment
 * M = sum_i q_i q_i^T (q [n][512]), by decreasing eigenvalue, each signed so that its entry of largest magnitude is
 * positive. With fewer queries than 512 the same vectors come from the n x n Gram matrix G[i][j] = q_i . q_j: an
 * eigenvector g of G with eigenvalue mu > 0 gives M's eigenvector sum_i g_i q_i / sqrt(mu), with the same eigenvalue
 * (M = Q^T Q and G = Q Q^T share their nonzero spectrum). eig receives the r_sk eigenvalues. Returns 0, or -1 when
 * r_sk is not in [1, 512] or the queries span fewer than r_sk directions. */
int vko_sketch_basis(const double* q, int64_t n, int32_t r_sk, double* vb, double* eig) {
  if (r_sk < 1 || r_sk > D_LAT || n < 1) return -1;
  const int gram = n < D_LAT;
  const int m = gram ? (int)n : D_LAT;
  if (r_sk > m) return -1;
  double* A = (double*)malloc(sizeof(double) * (size_t)m * m);
  double* ev = (double*)malloc(sizeof(double) * (size_t)m);
  double* vec = (double*)malloc(sizeof(double) * (size_t)m * m);
  if (gram) {
    for (int i = 0; i < m; ++i)
      for (int j = 0; j < m; ++j) {
        double acc = 0.0;
        for (int d = 0; d < D_LAT; ++d) acc += q[(int64_t)i * D_LAT + d] * q[(int64_t)j * D_LAT + d];
        A[i * m + j] = acc;
      }
  } else {
    for (int i = 0; i < m * m; ++i) A[i] = 0.0;
    for (int64_t t = 0; t < n; ++t)
      for (int i = 0; i < D_LAT; ++i)
        for (int j = 0; j < D_LAT; ++j) A[i * m + j] += q[t * D_LAT + i] * q[t * D_LAT + j];
  }
  jacobi_eig(m, A, ev, vec);
  int rc = 0;
  for (int k = 0; k < r_sk; ++k) {
    eig[k] = ev[k];
    double* out = vb + (int64_t)k * D_LAT;
    if (gram) {
      if (!(ev[k] > 0.0)) { rc = -1; break; }
      for (int d = 0; d < D_LAT; ++d) {
        double acc = 0.0;
        for (int i = 0; i < m; ++i) acc += vec[k * m + i] * q[(int64_t)i * D_LAT + d];
        out[d] = acc / sqrt(ev[k]);
      }
      int big = 0;
      for (int d = 1; d < D_LAT; ++d)
        if (fabs(out[d]) > fabs(out[big])) big = d;
      if (out[big] < 0.0)
        for (int d = 0; d < D_LAT; ++d) out[d] = -out[d];
    } else {
      for (int d = 0; d < D_LAT; ++d) out[d] = vec[k * m + d];
    }
  }
  free(vec);
  free(ev);
  free(A);
  return rc;
}

/* Index entry of every cached row: s_u = V_r^T L_u (s fp64 and s16 its bf16 RNE rounding, [B][N][r_sk], either may be
 * NULL) and eta_u = |L_u - V_r s_u| with the unrounded s_u ([B][N]). At r_sk = 0, eta_u = |L_u|. */
void vko_build_sketch(const vko_view* v, int32_t r_sk, const double* vb, double* s, uint16_t* s16, double* eta) {
  const int64_t N = v->N;
#pragma omp parallel for schedule(static)
  for (int b = 0; b < v->B; ++b) {
    double l[D_LAT], res[D_LAT];
    double* sk = (double*)malloc(sizeof(double) * (size_t)(r_sk > 0 ? r_sk : 1));
    for (int64_t u = 0; u < N; ++u) {
      for (int d = 0; d < D_LAT; ++d) { l[d] = L(v, b, u, d); res[d] = l[d]; }
      for (int j = 0; j < r_sk; ++j) {
        double acc = 0.0;
        for (int d = 0; d < D_LAT; ++d) acc += vb[(int64_t)j * D_LAT + d] * l[d];
        sk[j] = acc;
      }
      for (int j = 0; j < r_sk; ++j)
        for (int d = 0; d < D_LAT; ++d) res[d] -= sk[j] * vb[(int64_t)j * D_LAT + d];
      double e = 0.0;
      for (int d = 0; d < D_LAT; ++d) e += res[d] * res[d];
      eta[(int64_t)b * N + u] = sqrt(e);
      const int64_t o = ((int64_t)b * N + u) * r_sk;
      for (int j = 0; j < r_sk; ++j) {
        if (s) s[o + j] = sk[j];
        if (s16) s16[o + j] = vko_bf16_rne(sk[j]);
      }
    }
    free(sk);
  }
}

/* Query side of the sketch: p_h = V_r^T qc_h ([B][H][r_sk]) and rho_h = |qc_h - V_r p_h| ([B][H]). */
void vko_sketch_query(const vko_view* v, int32_t r_sk, const double* vb, double* p, double* rho) {
  for (int b = 0; b < v->B; ++b)
    for (int h = 0; h < v->H; ++h) {
      double q[D_LAT], res[D_LAT];
      const int64_t bh = (int64_t)b * v->H + h;
      for (int d = 0; d < D_LAT; ++d) { q[d] = QC(v, b, h, d); res[d] = q[d]; }
      for (int j = 0; j < r_sk; ++j) {
        double acc = 0.0;
        for (int d = 0; d < D_LAT; ++d) acc += vb[(int64_t)j * D_LAT + d] * q[d];
        p[bh * r_sk + j] = acc;
      }
      for (int j = 0; j < r_sk; ++j)
        for (int d = 0; d < D_LAT; ++d) res[d] -= p[bh * r_sk + j] * vb[(int64_t)j * D_LAT + d];
      double e = 0.0;
      for (int d = 0; d < D_LAT; ++d) e += res[d] * res[d];
      rho[bh] = sqrt(e);
    }
}

/* ---------------------------------------------------------------- conformal z (Sec. 4.2; Sec. 5) */
/* The trigger's certificate multiplier z from calibration queries. One recall target tau fixes the rest: the gate's
 * false-close budget alpha = (1 - tau)/2, the scan-level target tau_s = tau/(1 - alpha), the smallest calibration set
 * that can certify it min_hard = ceil(tau_s/(1 - tau_s)), and z = the ceil((n+1) tau_s)-th smallest required inflation
 * over n hard queries, clamped to Z_max. (Ceilings are taken 1e-9 below the exact value so that a ratio that is an
 * integer in exact arithmetic is not pushed up by rounding.) */
double vko_tau_s(double tau) {
  const double alpha = (1.0 - tau) / 2.0;
  return tau / (1.0 - alpha);
}

int64_t vko_min_hard(double tau) {
  const double ts = vko_tau_s(tau);
  return (int64_t)ceil(ts / (1.0 - ts) - 1e-9);
}

static int cmp_double(const void* x, const void* y) {
  const double a = *(const double*)x, b = *(const double*)y;
  return (a > b) - (a < b);
}

/* z from the required inflations zq[0, n) of the hard queries: Z_max when n < min_hard or the order statistic's
 * index exceeds n, else the k-th smallest (k = ceil((n+1) tau_s), 1-based); the result is clamped to [0, Z_max]. */
double vko_conformal_quantile(const double* zq, int64_t n, double tau, double z_max) {
  if (n < vko_min_hard(tau)) return z_max;
  const double x = (double)(n + 1) * vko_tau_s(tau);
  const int64_t k = (g_mutation == MUT_CONFORMAL_FLOOR) ? (int64_t)floor(x) : (int64_t)ceil(x - 1e-9);
  if (k > n || k < 1) return z_max;
  double* v = (double*)malloc(sizeof(double) * (size_t)n);
  for (int64_t i = 0; i < n; ++i) v[i] = zq[i];
  qsort(v, (size_t)n, sizeof(double), cmp_double);
  double z = v[k - 1];
  free(v);
  if (z > z_max) z = z_max;
  if (z < 0.0) z = 0.0;
  return z;
}

/* Every (b, h) is one calibration query. Its exact logits over all N cached rows give the causal argmax u* (ties: the
 * smaller position); the query is hard when u* lies outside its attended set S_h (idx/count), so that only the recall
 * tier can bring it back. For a hard query the required inflation is the z at which u*'s trigger score reaches the
 * tier-1 maximum s* = max over S_h: with sketch rank 0 the index part is idx_t = lambda (a[h,u*] +
 * |(O qr_h)[r:]| page_res[page(u*)]) and the certificate scale cert_t = lambda |qc_h| eta_u* / sqrt(d_c), d_c = 512,
 * so zq = (s* - idx_t) / cert_t. With a rank-r_sk content sketch (sk16, p, rho as for vko_trigger, eta the sketch
 * residual norms) the index part gains p_h . s_u* and the certificate is lambda rho_h eta_u* / sqrt(d_c - r_sk) (Eq. 4).
 * a, eta, page_res as from vko_scores and vko_build_index (or vko_build_sketch). zq[b,h] gets NaN for a query that
 * is not hard; ustar[b,h] the argmax row. Returns the number of hard queries. */
int64_t vko_calib_zq(const vko_view* v, int32_t r, const float* rot, double lam, const double* a, const double* eta,
                     const double* page_res, int32_t r_sk, const uint16_t* sk16, const double* p, const double* rho,
                     const int32_t* idx, const int32_t* count, int32_t cap, double* zq, int32_t* ustar) {
  const int64_t N = v->N, P = (N + PAGE - 1) / PAGE;
  int64_t n_hard = 0;
#pragma omp parallel for collapse(2) schedule(dynamic) reduction(+ : n_hard)
  for (int b = 0; b < v->B; ++b) {
    for (int h = 0; h < v->H; ++h) {
      const int64_t bh = (int64_t)b * v->H + h;
      char* in_set = (char*)calloc((size_t)N + 1, 1);
      int32_t n = count[bh];
      if (n > cap) n = cap;
      for (int32_t i = 0; i < n; ++i) in_set[idx[bh * cap + i]] = 1;
      double best = -INFINITY, sstar = -INFINITY;
      int64_t us = 0;
      for (int64_t u = 0; u < N; ++u) {
        const double s_u = logit(v, b, h, u, lam);
        if (s_u > best) { best = s_u; us = u; }
        if (in_set[u] && s_u > sstar) sstar = s_u;
      }
      ustar[bh] = (int32_t)us;
      if (in_set[us]) {
        zq[bh] = NAN;
      } else {
        double q[D_ROPE], qt[D_ROPE], qres = 0.0, qcn = 0.0;
        for (int j = 0; j < D_ROPE; ++j) q[j] = QR(v, b, h, j);
        if (r < D_ROPE) {
          rotate64(rot, q, qt);
          for (int j = r; j < D_ROPE; ++j) qres += qt[j] * qt[j];
          qres = sqrt(qres);
        }
        for (int j = 0; j < D_LAT; ++j) qcn += QC(v, b, h, j) * QC(v, b, h, j);
        qcn = sqrt(qcn);
        double skt = 0.0;
        for (int j = 0; j < r_sk; ++j) skt += p[bh * r_sk + j] * from_bf16(sk16[((int64_t)b * N + us) * r_sk + j]);
        const double idx_t = lam * (a[bh * N + us] + qres * page_res[(int64_t)b * P + us / PAGE] + skt);
        const double cq = r_sk > 0 ? rho[bh] : qcn;
        const double cert_t = lam * cq * eta[(int64_t)b * N + us] / sqrt((double)(D_LAT - r_sk));
        zq[bh] = (sstar - idx_t) / cert_t;
        ++n_hard;
      }
      free(in_set);
    }
  }
  return n_hard;
}

void vko_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

int vko_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
