/*
 * kvc_oracle.c -- plain, slow, fp64 CPU oracle for the decode step over a
 * sentinel-compressed KV cache (Ren et al., "Context Compression for
 * Auto-regressive Transformers with Sentinel Tokens", EMNLP 2023).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the
 * benchmark's CPU-baseline leg may load this library.  It shares no code,
 * header, table or helper with the CUDA path; every function below is written
 * from the paper's text, in the order the text states it, without blocking or
 * fusion.
 *
 * What it computes:
 *   - token positions with <CL>/<CR> tied to the previous token   (Sec. 3.1, Input Transformation)
 *   - the pairing of <CL> ... <CR> into non-overlapping spans     (Sec. 3.1, spans must not overlap)
 *   - the modified causal mask for one query                      (Sec. 1 and Sec. 3.1, Fig. 1 caption)
 *   - the rows that remain after the enclosed KV is freed         (Sec. 3.1, Manipulating Key-Value Memory)
 *   - single-query softmax attention over a set of rows, in fp64  (Sec. 2, Complexity of Attention)
 *   - RoPE (rotate-half convention) for the rotary configuration  (Sec. 1 cites rotary encoding; the
 *                                                                  convention is a reading, see below)
 *   - masked prefill: every query of a prompt block under the mask (Sec. 3.1)
 *   - the Local Attention baseline's window                       (Sec. 4.1 Baselines, Sec. 4.2)
 *
 * Readings of points the paper leaves open (each is also listed in the design notes):
 *   R1 <CL> is never visible to later queries under POLICY_PAPER (normal tokens see only "previous
 *      <CR> and normal tokens"); POLICY_KEEP_CL keeps and shows the <CL> row instead.
 *   R2 a <CR> query sees its own span's interior, earlier visible rows and itself, not <CL>.
 *   R3 a <CL> query sees itself only (stated explicitly in Sec. 3.1).
 *   R4 queries inside an open span see the earlier tokens of that span.
 *   R5 positions: a normal token takes the count of normal tokens before it; a sentinel takes the
 *      position of the token before it (0 at the start).  Positions are never renumbered.
 *   R6 RoPE: rotate-half on the first rotary_dim dims, theta_i = base^(-2i/rotary_dim); K is rotated
 *      at write time and the cache holds it rounded to the storage type; q is rotated at its own
 *      position and not rounded.
 *
 * Parity status: every function here is pinned by tests (brute force over all short kind sequences,
 * perturbation properties stated by the paper's mask rules, the compaction-equivalence invariant, a
 * library softmax-attention routine in the span-free case, closed-form counts, RoPE identities and
 * library float16/bfloat16 conversions).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORC_NORMAL = 0, ORC_CL = 1, ORC_CR = 2 };
enum { ORC_POLICY_PAPER = 0, ORC_POLICY_KEEP_CL = 1 };
enum { ORC_F16 = 0, ORC_BF16 = 1 };

#define ORC_OK 0
#define ORC_EINVAL (-1)
#define ORC_ESPAN (-2)
#define ORC_ENOMEM (-3)

/* ------------------------------------------------------------------------ */
/* 16-bit floating point, written from the IEEE 754 binary16 and the        */
/* bfloat16 (binary32 with the low 16 bits removed) formats.                */
/* ------------------------------------------------------------------------ */

double orc_f16_to_f64(uint16_t h) {
  int sign = (h >> 15) & 1;
  int ex = (h >> 10) & 0x1F;
  int man = h & 0x3FF;
  double v;
  if (ex == 0) {
    v = ldexp((double)man, -24); /* subnormal: man * 2^-24 */
  } else if (ex == 31) {
    v = man ? NAN : INFINITY;
  } else {
    v = ldexp((double)(man | 0x400), ex - 25); /* (1 + man/1024) * 2^(ex-15) */
  }
  return sign ? -v : v;
}

double orc_bf16_to_f64(uint16_t b) {
  int sign = (b >> 15) & 1;
  int ex = (b >> 7) & 0xFF;
  int man = b & 0x7F;
  double v;
  if (ex == 0) {
    v = ldexp((double)man, -133); /* subnormal: man * 2^(-126-7) */
  } else if (ex == 255) {
    v = man ? NAN : INFINITY;
  } else {
    v = ldexp((double)(man | 0x80), ex - 134); /* (1 + man/128) * 2^(ex-127) */
  }
  return sign ? -v : v;
}

/* Round x to a format with `mbits` stored significand bits, minimum normal exponent emin and
 * maximum exponent emax; nearest, ties to even.  Returns the encoded bits. */
static uint16_t orc_round_to_small(double x, int mbits, int emin, int emax, int ebias) {
  uint16_t sign = signbit(x) ? (uint16_t)(1u << 15) : 0;
  uint16_t inf_bits = (uint16_t)(((1u << (15 - mbits)) - 1u) << mbits);
  if (isnan(x)) return (uint16_t)(inf_bits | (1u << (mbits - 1)));
  double a = fabs(x);
  if (isinf(a)) return (uint16_t)(sign | inf_bits);
  if (a == 0.0) return sign;
  int e;
  (void)frexp(a, &e); /* a = f * 2^e with f in [0.5, 1) */
  e -= 1;             /* a = (2f) * 2^e, 2f in [1, 2) */
  if (e < emin) e = emin;
  double quantum = ldexp(1.0, e - mbits);
  double r = nearbyint(a / quantum); /* round-half-even in the default rounding mode */
  uint32_t one = 1u << mbits;
  if (r >= 2.0 * one) { /* carried into the next binade */
    r = one;
    e += 1;
  }
  if (e > emax) return (uint16_t)(sign | inf_bits);
  uint32_t ri = (uint32_t)r;
  if (ri < one) return (uint16_t)(sign | ri); /* subnormal (only possible at e == emin) */
  return (uint16_t)(sign | ((uint32_t)(e + ebias) << mbits) | (ri - one));
}

uint16_t orc_f64_to_f16(double x) { return orc_round_to_small(x, 10, -14, 15, 15); }
uint16_t orc_f64_to_bf16(double x) { return orc_round_to_small(x, 7, -126, 127, 127); }

static double orc_decode16(uint16_t v, int dtype) {
  return dtype == ORC_BF16 ? orc_bf16_to_f64(v) : orc_f16_to_f64(v);
}
static uint16_t orc_encode16(double x, int dtype) {
  return dtype == ORC_BF16 ? orc_f64_to_bf16(x) : orc_f64_to_f16(x);
}

void orc_decode16_array(int64_t n, const uint16_t* in, int dtype, double* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = orc_decode16(in[i], dtype);
}
void orc_encode16_array(int64_t n, const double* in, int dtype, uint16_t* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = orc_encode16(in[i], dtype);
}

/* ------------------------------------------------------------------------ */
/* Positions (Sec. 3.1, Input Transformation): <CL> and <CR> are tied to    */
/* the position of the token before them, so they occupy no position.      */
/* ------------------------------------------------------------------------ */

int orc_tied_positions(const uint8_t* kind, int64_t n, int32_t* pos) {
  int64_t normals_before = 0; /* normal tokens strictly before t */
  for (int64_t t = 0; t < n; ++t) {
    if (kind[t] > ORC_CR) return ORC_EINVAL;
    if (kind[t] == ORC_NORMAL) {
      pos[t] = (int32_t)normals_before; /* the next unused position */
      normals_before += 1;
    } else {
      pos[t] = t == 0 ? 0 : pos[t - 1]; /* tied to the previous token */
    }
  }
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Span pairing: each <CL> opens a span that the next <CR> closes; spans    */
/* must not overlap (Sec. 3.1), so a second <CL> inside an open span and a  */
/* <CR> without an open span are errors.                                     */
/* ------------------------------------------------------------------------ */

int orc_pair_spans(const uint8_t* kind, int64_t n, int64_t* cl, int64_t* cr, int64_t* n_closed, int64_t* open_cl) {
  int64_t open = -1, nc = 0;
  for (int64_t t = 0; t < n; ++t) {
    if (kind[t] == ORC_CL) {
      if (open >= 0) return ORC_ESPAN;
      open = t;
    } else if (kind[t] == ORC_CR) {
      if (open < 0) return ORC_ESPAN;
      if (cl) cl[nc] = open;
      if (cr) cr[nc] = t;
      nc += 1;
      open = -1;
    } else if (kind[t] != ORC_NORMAL) {
      return ORC_EINVAL;
    }
  }
  *n_closed = nc;
  *open_cl = open;
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* The modified causal mask for the query at index t_q (Sec. 1; Sec. 3.1):  */
/*  - <CL> attends only to itself;                                          */
/*  - other tokens attend to earlier <CR> and normal tokens, except that     */
/*    tokens after a <CR> may not attend to the tokens between that span's   */
/*    <CL> and <CR>.                                                         */
/* vis[j] for j in [0, t_q].                                                 */
/* ------------------------------------------------------------------------ */

int orc_visible(const uint8_t* kind, int64_t t_q, int policy, uint8_t* vis) {
  if (t_q < 0) return ORC_EINVAL;
  int64_t n = t_q + 1;
  int64_t* cl = (int64_t*)malloc(sizeof(int64_t) * (size_t)(n / 2 + 1));
  int64_t* cr = (int64_t*)malloc(sizeof(int64_t) * (size_t)(n / 2 + 1));
  if (!cl || !cr) {
    free(cl);
    free(cr);
    return ORC_ENOMEM;
  }
  int64_t nc = 0, open = -1;
  int rc = orc_pair_spans(kind, n, cl, cr, &nc, &open);
  if (rc != ORC_OK) {
    free(cl);
    free(cr);
    return rc;
  }
  for (int64_t j = 0; j <= t_q; ++j) {
    if (kind[t_q] == ORC_CL) { /* R3 */
      vis[j] = (uint8_t)(j == t_q);
      continue;
    }
    int v = 1;
    if (kind[j] == ORC_CL && policy == ORC_POLICY_PAPER) v = 0; /* R1 */
    for (int64_t k = 0; k < nc; ++k) {
      if (cr[k] < t_q && cl[k] < j && j < cr[k]) v = 0; /* strictly inside a span closed before t_q */
    }
    vis[j] = (uint8_t)v;
  }
  free(cl);
  free(cr);
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Freeing the enclosed KV (Sec. 3.1, Manipulating Key-Value Memory): the    */
/* rows kept from a history of n_hist tokens after the given spans are       */
/* freed.  POLICY_PAPER frees <CL> and the interior, POLICY_KEEP_CL only     */
/* the interior; <CR> is always kept.  rows[] is increasing.                 */
/* ------------------------------------------------------------------------ */

int orc_stored_rows(int64_t n_hist, const int64_t* cl, const int64_t* cr, int64_t n_spans, int policy, int64_t* rows,
                    int64_t* n_rows) {
  int64_t n = 0;
  for (int64_t j = 0; j < n_hist; ++j) {
    int keep = 1;
    for (int64_t k = 0; k < n_spans; ++k) {
      int64_t lo = policy == ORC_POLICY_PAPER ? cl[k] : cl[k] + 1;
      if (lo <= j && j < cr[k]) keep = 0;
    }
    if (keep) rows[n++] = j;
  }
  *n_rows = n;
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* RoPE, rotate-half convention (reading R6).                                */
/* ------------------------------------------------------------------------ */

void orc_rope(const double* x, int d, int rot, double base, double pos, double* y) {
  int half = rot / 2;
  for (int i = 0; i < d; ++i) y[i] = x[i];
  for (int i = 0; i < half; ++i) {
    double theta = pos * pow(base, -2.0 * (double)i / (double)rot);
    double c = cos(theta), s = sin(theta);
    y[i] = x[i] * c - x[i + half] * s;
    y[i + half] = x[i + half] * c + x[i] * s;
  }
}

/* ------------------------------------------------------------------------ */
/* Single-query softmax attention over an explicit set of rows (Sec. 2):      */
/*   z_j = scale * <q', k'_j>,  out = sum_j softmax(z)_j v_j                   */
/* K, V: [n_hist][d] 16-bit bits of one (sequence, head); rows: indices into  */
/* them; pos: per-row positions (RoPE only); qpos: the query's position.      */
/* ------------------------------------------------------------------------ */

int orc_attend(int d, int dtype, const uint16_t* q, const uint16_t* K, const uint16_t* V, const int32_t* pos,
               const int64_t* rows, int64_t n_rows, double scale, int rot, double base, int32_t qpos, double* out) {
  if (n_rows <= 0) return ORC_EINVAL;
  double* qv = (double*)malloc(sizeof(double) * (size_t)d * 4);
  double* z = (double*)malloc(sizeof(double) * (size_t)n_rows);
  if (!qv || !z) {
    free(qv);
    free(z);
    return ORC_ENOMEM;
  }
  double* qr = qv + d;
  double* kv = qv + 2 * d;
  double* kr = qv + 3 * d;
  for (int e = 0; e < d; ++e) qv[e] = orc_decode16(q[e], dtype);
  if (rot > 0) {
    orc_rope(qv, d, rot, base, (double)qpos, qr);
  } else {
    for (int e = 0; e < d; ++e) qr[e] = qv[e];
  }
  for (int64_t r = 0; r < n_rows; ++r) {
    const uint16_t* krow = K + rows[r] * (int64_t)d;
    for (int e = 0; e < d; ++e) kv[e] = orc_decode16(krow[e], dtype);
    if (rot > 0) {
      /* the cache holds K rotated at its own position, rounded to the storage type (R6) */
      orc_rope(kv, d, rot, base, (double)pos[rows[r]], kr);
      for (int e = 0; e < d; ++e) kr[e] = orc_decode16(orc_encode16(kr[e], dtype), dtype);
    } else {
      for (int e = 0; e < d; ++e) kr[e] = kv[e];
    }
    double dot = 0.0;
    for (int e = 0; e < d; ++e) dot += qr[e] * kr[e];
    z[r] = scale * dot;
  }
  double m = -INFINITY;
  for (int64_t r = 0; r < n_rows; ++r)
    if (z[r] > m) m = z[r];
  double l = 0.0;
  for (int64_t r = 0; r < n_rows; ++r) {
    z[r] = exp(z[r] - m);
    l += z[r];
  }
  for (int e = 0; e < d; ++e) out[e] = 0.0;
  for (int64_t r = 0; r < n_rows; ++r) {
    const uint16_t* vrow = V + rows[r] * (int64_t)d;
    double p = z[r] / l;
    for (int e = 0; e < d; ++e) out[e] += p * orc_decode16(vrow[e], dtype);
  }
  free(qv);
  free(z);
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* The decode step under the modified mask over the FULL (never compacted)   */
/* history, for a batch of sequences and heads.  The query of sequence s is  */
/* its last token, t_q = n_hist[s] - 1, at position pos[t_q].                */
/*   kinds/pos: histories concatenated, sequence s at hist_off[s]            */
/*   K/V: [H][n_hist[s]][d] of sequence s at element offset kv_off[s]        */
/*   q:   [n_seq][H][d];  out: [n_seq][H][d] (fp64)                          */
/* Heads are independent; H may be any subset of a model's heads.           */
/* ------------------------------------------------------------------------ */

int orc_masked_decode(int64_t n_seq, int64_t H, int d, int dtype, const int64_t* n_hist, const int64_t* hist_off,
                      const uint8_t* kinds, const int32_t* pos, const int64_t* kv_off, const uint16_t* K,
                      const uint16_t* V, const uint16_t* q, double scale, int rot, double base, int policy,
                      double* out, int n_threads) {
  int rc_all = ORC_OK;
  int64_t** rows = (int64_t**)calloc((size_t)n_seq, sizeof(int64_t*));
  int64_t* n_rows = (int64_t*)calloc((size_t)n_seq, sizeof(int64_t));
  if (!rows || !n_rows) {
    free(rows);
    free(n_rows);
    return ORC_ENOMEM;
  }
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#else
  (void)n_threads;
#endif
  /* the visible set of each sequence's query (shared by its heads) */
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t s = 0; s < n_seq; ++s) {
    int64_t t_q = n_hist[s] - 1;
    uint8_t* vis = (uint8_t*)malloc((size_t)(t_q + 1));
    rows[s] = (int64_t*)malloc(sizeof(int64_t) * (size_t)(t_q + 1));
    if (!vis || !rows[s]) {
#pragma omp atomic write
      rc_all = ORC_ENOMEM;
      free(vis);
      continue;
    }
    int rc = orc_visible(kinds + hist_off[s], t_q, policy, vis);
    if (rc != ORC_OK) {
#pragma omp atomic write
      rc_all = rc;
    }
    int64_t n = 0;
    for (int64_t j = 0; j <= t_q; ++j)
      if (vis[j]) rows[s][n++] = j;
    n_rows[s] = n;
    free(vis);
  }
  if (rc_all == ORC_OK) {
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t sh = 0; sh < n_seq * H; ++sh) {
      int64_t s = sh / H, h = sh % H;
      int64_t T = n_hist[s];
      const uint16_t* Ks = K + kv_off[s] + h * T * d;
      const uint16_t* Vs = V + kv_off[s] + h * T * d;
      const int32_t* ps = pos + hist_off[s];
      int rc = orc_attend(d, dtype, q + (s * H + h) * d, Ks, Vs, ps, rows[s], n_rows[s], scale, rot, base,
                          ps[T - 1], out + (s * H + h) * d);
      if (rc != ORC_OK) {
#pragma omp atomic write
        rc_all = rc;
      }
    }
  }
  for (int64_t s = 0; s < n_seq; ++s) free(rows[s]);
  free(rows);
  free(n_rows);
  return rc_all;
}

int orc_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* ------------------------------------------------------------------------ */
/* Local Attention baseline (Sec. 4.1 Baselines; Sec. 4.2: a FIFO queue of   */
/* key-value memory at inference): token x_t (1-based t) attends within      */
/* (floor(t*r), t].  With 0-based history indices, the query at index t_q     */
/* sees j = floor((t_q + 1) * r) .. t_q (reading R14: the window closes on    */
/* the query itself, as every causal mask does).                             */
/* ------------------------------------------------------------------------ */

int orc_visible_local(int64_t t_q, double ratio, uint8_t* vis) {
  if (t_q < 0 || !(ratio >= 0.0) || !(ratio < 1.0)) return ORC_EINVAL;
  const int64_t first = (int64_t)floor((double)(t_q + 1) * ratio); /* first visible index */
  for (int64_t j = 0; j <= t_q; ++j) vis[j] = (uint8_t)(j >= first);
  return ORC_OK;
}

/* Decode under the Local Attention mask over full histories (layout as orc_masked_decode). */
int orc_local_decode(int64_t n_seq, int64_t H, int d, int dtype, const int64_t* n_hist, const int64_t* hist_off,
                     const int32_t* pos, const int64_t* kv_off, const uint16_t* K, const uint16_t* V,
                     const uint16_t* q, double scale, int rot, double base, double ratio, double* out,
                     int n_threads) {
  int rc_all = ORC_OK;
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#else
  (void)n_threads;
#endif
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t sh = 0; sh < n_seq * H; ++sh) {
    int64_t s = sh / H, h = sh % H;
    int64_t T = n_hist[s];
    uint8_t* vis = (uint8_t*)malloc((size_t)T);
    int64_t* rows = (int64_t*)malloc(sizeof(int64_t) * (size_t)T);
    int rc = (vis && rows) ? orc_visible_local(T - 1, ratio, vis) : ORC_ENOMEM;
    if (rc == ORC_OK) {
      int64_t n = 0;
      for (int64_t j = 0; j < T; ++j)
        if (vis[j]) rows[n++] = j;
      const int32_t* ps = pos + hist_off[s];
      rc = orc_attend(d, dtype, q + (s * H + h) * d, K + kv_off[s] + h * T * d, V + kv_off[s] + h * T * d, ps, rows,
                      n, scale, rot, base, ps[T - 1], out + (s * H + h) * d);
    }
    if (rc != ORC_OK) {
#pragma omp atomic write
      rc_all = rc;
    }
    free(vis);
    free(rows);
  }
  return rc_all;
}

/* ------------------------------------------------------------------------ */
/* Masked prefill (Sec. 3.1: the modified mask holds for every token of a    */
/* prompt in the forward pass; Manipulating Key-Value Memory: a long prefix  */
/* may be run block by block).  For sequence s the queries are its last      */
/* n_q[s] history tokens; the query at history index t attends to [0, t]     */
/* under orc_visible(t) -- the same rows a decode step at t would see.       */
/*   kinds/pos/K/V: as orc_masked_decode                                     */
/*   Q:   [sum n_q][H][d], sequence s's queries from row q_off[s], oldest    */
/*        first; out: same layout, fp64.                                     */
/* ------------------------------------------------------------------------ */

int orc_masked_prefill(int64_t n_seq, int64_t H, int d, int dtype, const int64_t* n_hist, const int64_t* hist_off,
                       const uint8_t* kinds, const int32_t* pos, const int64_t* kv_off, const uint16_t* K,
                       const uint16_t* V, const int64_t* n_q, const int64_t* q_off, const uint16_t* Q,
                       double scale, int rot, double base, int policy, double* out, int n_threads) {
  int64_t n_items = 0;
  for (int64_t s = 0; s < n_seq; ++s) {
    if (n_q[s] < 0 || n_q[s] > n_hist[s]) return ORC_EINVAL;
    n_items += n_q[s];
  }
  int rc_all = ORC_OK;
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#else
  (void)n_threads;
#endif
#pragma omp parallel for schedule(dynamic, 4)
  for (int64_t it = 0; it < n_items; ++it) {
    /* item -> (sequence, query) by a linear walk: plain, and cheap beside the attention */
    int64_t s = 0, i = it;
    while (i >= n_q[s]) i -= n_q[s++];
    const int64_t T = n_hist[s];
    const int64_t t = T - n_q[s] + i; /* the query's history index */
    uint8_t* vis = (uint8_t*)malloc((size_t)(t + 1));
    int64_t* rows = (int64_t*)malloc(sizeof(int64_t) * (size_t)(t + 1));
    int rc = (vis && rows) ? orc_visible(kinds + hist_off[s], t, policy, vis) : ORC_ENOMEM;
    if (rc == ORC_OK) {
      int64_t n = 0;
      for (int64_t j = 0; j <= t; ++j)
        if (vis[j]) rows[n++] = j;
      const int32_t* ps = pos + hist_off[s];
      for (int64_t h = 0; h < H && rc == ORC_OK; ++h) {
        const int64_t qrow = (q_off[s] + i) * H + h;
        rc = orc_attend(d, dtype, Q + qrow * d, K + kv_off[s] + h * T * d, V + kv_off[s] + h * T * d, ps, rows, n,
                        scale, rot, base, ps[t], out + qrow * d);
      }
    }
    if (rc != ORC_OK) {
#pragma omp atomic write
      rc_all = rc;
    }
    free(vis);
    free(rows);
  }
  return rc_all;
}
