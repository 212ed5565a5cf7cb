/*
 * akv_oracle.c -- plain, slow, fp64 CPU oracle of AnchorKV (arXiv 2608.02901).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path links, loads or
 * calls this file; only the tests, the smoke check and the CPU-baseline leg
 * of the benchmark do.  It shares no code, header, table or constant
 * generator with the CUDA library: every formula below is written from the
 * paper (and from the readings recorded where the paper is silent).
 *
 * What it computes
 *   encode  : Section 3.1 Eq. 1 (absolute-cosine nearest anchor), Eq. 2
 *             (projection coefficient, residual), Section 3.2 (last W
 *             positions are anchors, the rest sampled uniformly), Appendix
 *             A.1 Eq. 12 (randomized Hadamard rotation) and a 4-level
 *             2-bit quantizer: uniform with per-token fp16 scale and min, or
 *             the Lloyd-Max codebook of Section 3.1 with a per-token RMS
 *             scale; residual
 *             slots ranked by residual norm (Section 4.3, variant (ii)).
 *   encode_select : Algorithm 1 with the paper's full selection: the last W
 *             positions, a share rho of the other anchors by the selector
 *             score of Appendix A.2 (observation queries' attention, average
 *             pooled over kappa positions), the rest sampled uniformly; the
 *             output-aware utilities of Eq. 6; the layer budget of Eq. 9
 *             (Appendix A.1 accounting) split floor(N/2) keys, the rest
 *             values, each side's top-N pooled over the layer's KV heads.
 *   attend  : Eq. 3 reconstruction of every key and value, then Eq. 4
 *             softmax attention, all in fp64, one token at a time; with an
 *             exact dense suffix (Appendix E.1 and E.2: generated tokens kept
 *             in bf16) the suffix tokens join the same softmax; with RoPE at
 *             decode (Section 3.2) every key is turned to its position first.
 *   attend_factorized : the same attention regrouped by anchor (anchor
 *             scores computed once, value weights summed per anchor, inverse
 *             rotation applied once after accumulation -- Section 4.4 and
 *             Appendix E.1 rely on this linearity); used only to pin that
 *             regrouping against the definition.
 *   unpack  : an independent reader of the packed arena layout (tile blocks,
 *             tokens in the arena's stored order).
 *
 * Compiled with -ffp-contract=off so that every product and sum is the
 * separately rounded IEEE operation written here.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_D 128
/* Codec flags (the library's AKV_FLAG_ROTATE and AKV_FLAG_LLOYD bits). */
#define OR_ROTATE 1
#define OR_LLOYD 2
#define OR_ROPE 4

/* The four-level Lloyd-Max quantizer of a unit Gaussian source (Max 1960, the
 * codebook of Section 3.1 and Appendix A.1): levels -1.5104, -0.4528, 0.4528,
 * 1.5104, decision thresholds at their midpoints.  The levels are taken to 8
 * significant bits (+-0.453125, +-1.5078125: exact in bf16 and fp16, so the
 * decoder's tensor-core operands carry them unrounded) and the thresholds are
 * the midpoints of those levels (0, +-0.98046875). */
static const double OR_LM_LEVEL[4] = {-1.5078125, -0.453125, 0.453125, 1.5078125};
#define OR_LM_T 0.98046875

/* Reconstruction value of a 2-bit code: the code itself (uniform codec) or its
 * Lloyd-Max level. */
static double or_level(int flags, int c) { return (flags & OR_LLOYD) ? OR_LM_LEVEL[c] : (double)c; }

/* ------------------------------------------------------------------------ */
/* Scalar helpers                                                            */
/* ------------------------------------------------------------------------ */

/* SplitMix64 output function (Steele, Lea and Flood, OOPSLA 2014): the state
 * advanced by the golden-ratio increment, then the 64-bit finaliser. */
uint64_t or_splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

/* bf16 bits -> exact double. */
double or_bf16_to_double(uint16_t b) {
  uint32_t u = ((uint32_t)b) << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

/* fp16 bits -> exact double. */
double or_fp16_to_double(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 10) & 0x1F;
  int m = h & 0x3FF;
  double v;
  if (e == 0) {
    v = ldexp((double)m, -24);
  } else if (e == 31) {
    v = m ? NAN : INFINITY;
  } else {
    v = ldexp((double)(1024 + m), e - 25);
  }
  return sign ? -v : v;
}

/* double -> fp16 bits, round to nearest even, saturating at +-65504.
 * Direct from the double value (no float intermediate). */
uint16_t or_fp16_from_double(double x) {
  if (isnan(x)) return 0x7E00;
  uint16_t sign = signbit(x) ? 0x8000 : 0;
  double a = fabs(x);
  if (a >= 65504.0) return (uint16_t)(sign | 0x7BFF);
  if (a < ldexp(1.0, -14)) {
    /* subnormal range: integer multiples of 2^-24 */
    double r = rint(a * 16777216.0);
    return (uint16_t)(sign | (uint16_t)r);
  }
  int e;
  double m = frexp(a, &e); /* a = m 2^e, m in [0.5, 1) */
  double frac = (2.0 * m - 1.0) * 1024.0;
  double r = rint(frac);
  uint32_t bits = ((uint32_t)(e + 14) << 10) + (uint32_t)r;
  if (bits >= 0x7C00) bits = 0x7BFF;
  return (uint16_t)(sign | bits);
}

/* Rotation signs s_j (Appendix A.1, Eq. 12): bit (j mod 64) of
 * splitmix64(rot_seed + floor(j / 64)); a set bit means -1. */
void or_signs(uint64_t rot_seed, double* s) {
  for (int j = 0; j < OR_D; ++j) {
    uint64_t w = or_splitmix64(rot_seed + (uint64_t)(j / 64));
    s[j] = ((w >> (j % 64)) & 1ull) ? -1.0 : 1.0;
  }
}

/* In-place unnormalised Walsh-Hadamard transform of length 128 in Sylvester
 * (natural) order: stages h = 1, 2, ..., 64, pairs (a, b) -> (a + b, a - b). */
void or_wht128(double* v) {
  for (int h = 1; h < OR_D; h <<= 1) {
    for (int i = 0; i < OR_D; i += 2 * h) {
      for (int j = i; j < i + h; ++j) {
        double a = v[j], b = v[j + h];
        v[j] = a + b;
        v[j + h] = a - b;
      }
    }
  }
}

/* ------------------------------------------------------------------------ */
/* Shapes (Section 3.2 anchor budget incl. the window; residual budgets)     */
/* ------------------------------------------------------------------------ */

void or_unit_shape(int32_t S, float f_a, float f_rk, float f_rv, int32_t W, int32_t* k, int32_t* nk,
                   int32_t* nv) {
  int32_t w = W < S ? W : S;
  double ka = ceil((double)f_a * (double)S);
  int32_t kk = (int32_t)ka;
  if (kk < w) kk = w;
  if (kk > S) kk = S;
  int32_t rk = (int32_t)floor((double)f_rk * (double)S);
  int32_t rv = (int32_t)floor((double)f_rv * (double)S);
  if (rk > S - kk) rk = S - kk;
  if (rv > S - kk) rv = S - kk;
  *k = kk;
  *nk = rk;
  *nv = rv;
}

/* ------------------------------------------------------------------------ */
/* One unit's logical compressed cache                                       */
/* ------------------------------------------------------------------------ */

typedef struct or_unit {
  int32_t S, k, nk, nv;
  uint16_t* anchor_k;  /* [k][128] bf16 */
  uint16_t* anchor_v;  /* [k][128] bf16 */
  int32_t* anchor_pos; /* [k] */
  uint16_t* idx_k;     /* [S] */
  uint16_t* gam_k;     /* [S] fp16 */
  uint16_t* idx_v;
  uint16_t* gam_v;
  int32_t* res_k; /* [nk] ascending positions */
  uint8_t* codes_k; /* [nk][32] */
  uint16_t* scale_k; /* [nk] fp16 */
  uint16_t* min_k;   /* [nk] fp16 */
  int32_t* res_v;
  uint8_t* codes_v;
  uint16_t* scale_v;
  uint16_t* min_v;
  int32_t* pos; /* [S] position of index i (RoPE at decode); NULL: position i */
} or_unit;

typedef struct {
  uint64_t key;
  int32_t pos;
} or_keypos;

static int cmp_key_asc(const void* a, const void* b) {
  const or_keypos* x = (const or_keypos*)a;
  const or_keypos* y = (const or_keypos*)b;
  if (x->key < y->key) return -1;
  if (x->key > y->key) return 1;
  return (x->pos < y->pos) ? -1 : (x->pos > y->pos);
}

typedef struct {
  double e;
  int32_t pos;
} or_errpos;

/* larger residual energy first; equal energies: lower position first */
static int cmp_err_desc(const void* a, const void* b) {
  const or_errpos* x = (const or_errpos*)a;
  const or_errpos* y = (const or_errpos*)b;
  if (x->e > y->e) return -1;
  if (x->e < y->e) return 1;
  return (x->pos < y->pos) ? -1 : (x->pos > y->pos);
}

static int cmp_i32(const void* a, const void* b) {
  int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
  return (x > y) - (x < y);
}

/* Quantize one residual and pack 4 codes per byte (code j in byte j/4, bits
 * 2(j%4)..+1).  Appendix A.1 rotation first (v = H(s o r), when flags has
 * OR_ROTATE), then one of two codecs:
 *   uniform  : 4-level uniform codes on [min, max] with fp16 scale and min,
 *              c^_j = min + code_j scale;
 *   Lloyd-Max: (OR_LLOYD) each coordinate divided by the per-token RMS scale
 *              sigma = sqrt(sum_j v_j^2 / 128) (the rotated coordinates are
 *              about N(0, sigma^2), Appendix A.1; the sum taken in index
 *              order), fp16 scale, min 0, code = the Lloyd-Max decision region
 *              of v_j / scale, c^_j = scale L[code]. */
static void or_quantize(const double* r, const double* s, int flags, uint8_t* codes, uint16_t* sc_out,
                        uint16_t* mn_out) {
  double v[OR_D];
  for (int j = 0; j < OR_D; ++j) v[j] = (flags & OR_ROTATE) ? s[j] * r[j] : r[j];
  if (flags & OR_ROTATE) or_wht128(v);
  memset(codes, 0, 32);
  if (flags & OR_LLOYD) {
    double ss = 0.0;
    for (int j = 0; j < OR_D; ++j) ss += v[j] * v[j];
    uint16_t sc_h = or_fp16_from_double(sqrt(ss / (double)OR_D));
    double sc = or_fp16_to_double(sc_h);
    for (int j = 0; j < OR_D; ++j) {
      int c = 2; /* a zero scale: every level reconstructs 0 */
      if (sc != 0.0) {
        double t = v[j] / sc;
        c = t < -OR_LM_T ? 0 : (t < 0.0 ? 1 : (t < OR_LM_T ? 2 : 3));
      }
      codes[j / 4] |= (uint8_t)(c << (2 * (j % 4)));
    }
    *sc_out = sc_h;
    *mn_out = 0;
    return;
  }
  double vmin = v[0], vmax = v[0];
  for (int j = 1; j < OR_D; ++j) {
    if (v[j] < vmin) vmin = v[j];
    if (v[j] > vmax) vmax = v[j];
  }
  uint16_t mn_h = or_fp16_from_double(vmin);
  double mn = or_fp16_to_double(mn_h);
  double t = (vmax - mn) / 3.0;
  if (!(t > 0.0)) t = 0.0;
  uint16_t sc_h = or_fp16_from_double(t);
  double sc = or_fp16_to_double(sc_h);
  for (int j = 0; j < OR_D; ++j) {
    int c = 0;
    if (sc != 0.0) {
      double q = rint((v[j] - mn) / sc);
      if (q < 0.0) q = 0.0;
      if (q > 3.0) q = 3.0;
      c = (int)q;
    }
    codes[j / 4] |= (uint8_t)(c << (2 * (j % 4)));
  }
  *sc_out = sc_h;
  *mn_out = mn_h;
}

/* Exported for the quantizer pins: rotate (if set) and quantize one residual r[128]. */
void or_quantize_residual(const double* r, uint64_t rot_seed, int flags, uint8_t* codes, uint16_t* sc,
                          uint16_t* mn) {
  double s[OR_D];
  or_signs(rot_seed, s);
  or_quantize(r, s, flags, codes, sc, mn);
}

/* Encode one side (keys or values) of one unit given the anchor set. */
static void or_encode_side(int32_t S, int32_t k, int32_t nres, const uint16_t* X /*[S][128]*/,
                           const int32_t* anchor_pos, const int32_t* slot_of, const double* s, int flags,
                           uint16_t* idx, uint16_t* gam, int32_t* res, uint8_t* codes, uint16_t* scale,
                           uint16_t* mins) {
  /* anchor rows as doubles (exact) and their squared norms */
  double* n = (double*)malloc(sizeof(double) * (size_t)(k > 0 ? k : 1));
  double* xad = (double*)malloc(sizeof(double) * (size_t)(k > 0 ? k : 1) * OR_D);
  for (int32_t a = 0; a < k; ++a) {
    const uint16_t* xa = X + (size_t)anchor_pos[a] * OR_D;
    double acc = 0.0;
    for (int j = 0; j < OR_D; ++j) {
      double t = or_bf16_to_double(xa[j]);
      xad[(size_t)a * OR_D + j] = t;
      acc = acc + t * t;
    }
    n[a] = acc;
  }
  or_errpos* cand = (or_errpos*)malloc(sizeof(or_errpos) * (size_t)(S > 0 ? S : 1));
  int32_t ncand = 0;
  double xi[OR_D], r[OR_D];
  for (int32_t i = 0; i < S; ++i) {
    if (slot_of[i] >= 0) { /* anchors are exact: own slot, gamma = 1 */
      idx[i] = (uint16_t)slot_of[i];
      gam[i] = 0x3C00;
      continue;
    }
    const uint16_t* x = X + (size_t)i * OR_D;
    for (int j = 0; j < OR_D; ++j) xi[j] = or_bf16_to_double(x[j]);
    /* Eq. 1: largest |<x_i, x_a>| / ||x_a|| (||x_i|| is common to all a). */
    int32_t best = -1;
    double bestc = -1.0, bestd = 0.0;
    for (int32_t a = 0; a < k; ++a) {
      if (n[a] == 0.0) continue;
      const double* xa = xad + (size_t)a * OR_D;
      double d = 0.0;
      for (int j = 0; j < OR_D; ++j) d = d + xi[j] * xa[j];
      double c = fabs(d) / sqrt(n[a]);
      if (c > bestc) {
        bestc = c;
        best = a;
        bestd = d;
      }
    }
    uint16_t g_h = 0;
    if (best >= 0) g_h = or_fp16_from_double(bestd / n[best]); /* Eq. 2 */
    idx[i] = (uint16_t)(best >= 0 ? best : 0);
    gam[i] = g_h;
    /* Eq. 2 residual with the stored coefficient, and its energy */
    double g = or_fp16_to_double(g_h);
    const uint16_t* xa = X + (size_t)anchor_pos[best >= 0 ? best : 0] * OR_D;
    double e = 0.0;
    for (int j = 0; j < OR_D; ++j) {
      double p = (best >= 0) ? g * or_bf16_to_double(xa[j]) : 0.0;
      double rj = xi[j] - p;
      e = e + rj * rj;
    }
    cand[ncand].e = e;
    cand[ncand].pos = i;
    ++ncand;
  }
  /* residual slots: the nres largest energies among non-anchors */
  qsort(cand, (size_t)ncand, sizeof(or_errpos), cmp_err_desc);
  for (int32_t t = 0; t < nres; ++t) res[t] = cand[t].pos;
  if (nres > 0) qsort(res, (size_t)nres, sizeof(int32_t), cmp_i32);
  for (int32_t t = 0; t < nres; ++t) {
    int32_t i = res[t];
    const uint16_t* x = X + (size_t)i * OR_D;
    const uint16_t* xa = X + (size_t)anchor_pos[idx[i]] * OR_D;
    double g = or_fp16_to_double(gam[i]);
    int valid = 0;
    for (int32_t a = 0; a < k; ++a)
      if (n[a] != 0.0) valid = 1;
    for (int j = 0; j < OR_D; ++j) {
      double p = valid ? g * or_bf16_to_double(xa[j]) : 0.0;
      r[j] = or_bf16_to_double(x[j]) - p;
    }
    or_quantize(r, s, flags, codes + (size_t)t * 32, &scale[t], &mins[t]);
  }
  free(cand);
  free(xad);
  free(n);
}

/*
 * Encode one (request b, KV head h) unit.  K and V are bf16 bits [S][128].
 * The caller allocates every array of `u` with the sizes of or_unit_shape
 * and sets u->S, k, nk, nv.
 */
int or_encode_unit(const uint16_t* K, const uint16_t* V, int32_t b, int32_t h, int32_t W, uint64_t seed,
                   uint64_t rot_seed, int flags, or_unit* u) {
  int32_t S = u->S, k = u->k;
  int32_t w = W < S ? W : S;
  /* Section 3.2: the last w positions are anchors; the k - w others are a
   * uniform sample of [0, S - w): the positions with the smallest hash. */
  int32_t* slot_of = (int32_t*)malloc(sizeof(int32_t) * (size_t)S);
  char* is_anchor = (char*)calloc((size_t)S, 1);
  int32_t rest = k - w;
  if (rest > 0) {
    int32_t pool = S - w;
    or_keypos* kp = (or_keypos*)malloc(sizeof(or_keypos) * (size_t)pool);
    uint64_t base = seed ^ ((uint64_t)b << 40) ^ ((uint64_t)h << 32);
    for (int32_t p = 0; p < pool; ++p) {
      kp[p].key = or_splitmix64(base ^ (uint64_t)p);
      kp[p].pos = p;
    }
    qsort(kp, (size_t)pool, sizeof(or_keypos), cmp_key_asc);
    for (int32_t t = 0; t < rest; ++t) is_anchor[kp[t].pos] = 1;
    free(kp);
  }
  for (int32_t p = S - w; p < S; ++p) is_anchor[p] = 1;
  int32_t t = 0;
  for (int32_t p = 0; p < S; ++p) {
    if (is_anchor[p]) {
      u->anchor_pos[t] = p;
      slot_of[p] = t;
      ++t;
    } else {
      slot_of[p] = -1;
    }
  }
  if (t != k) {
    free(slot_of);
    free(is_anchor);
    return -1;
  }
  for (int32_t a = 0; a < k; ++a) {
    memcpy(u->anchor_k + (size_t)a * OR_D, K + (size_t)u->anchor_pos[a] * OR_D, OR_D * 2);
    memcpy(u->anchor_v + (size_t)a * OR_D, V + (size_t)u->anchor_pos[a] * OR_D, OR_D * 2);
  }
  double s[OR_D];
  or_signs(rot_seed, s);
  or_encode_side(S, k, u->nk, K, u->anchor_pos, slot_of, s, flags, u->idx_k, u->gam_k, u->res_k, u->codes_k,
                 u->scale_k, u->min_k);
  or_encode_side(S, k, u->nv, V, u->anchor_pos, slot_of, s, flags, u->idx_v, u->gam_v, u->res_v, u->codes_v,
                 u->scale_v, u->min_v);
  free(slot_of);
  free(is_anchor);
  return 0;
}

/* Batched encode: K, V are [n_units][s_max][128]; units[u] describe b = u / H, h = u % H. */
int or_encode_batch(const uint16_t* K, const uint16_t* V, int32_t s_max, int32_t n_units, int32_t H, int32_t W,
                    uint64_t seed, uint64_t rot_seed, int flags, or_unit* units) {
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
  for (int32_t u = 0; u < n_units; ++u) {
    size_t off = (size_t)u * (size_t)s_max * OR_D;
    if (or_encode_unit(K + off, V + off, u / H, u % H, W, seed, rot_seed, flags, &units[u]) != 0) bad |= 1;
  }
  return bad ? -1 : 0;
}

/* ------------------------------------------------------------------------ */
/* Reconstruction (Eq. 3) and attention (Eq. 4)                              */
/* ------------------------------------------------------------------------ */

/* r~ = U^T C^{-1}(q) of Eq. 14 with U = H diag(s) / sqrt(D): here the stored
 * codes dequantize to c^ = min + L(code) * scale in the sqrt(D)-scaled rotated
 * domain (L(code) = code, or the Lloyd-Max level), so r~ = s o (H c^) / D. */
static void or_dequant_residual(const uint8_t* codes, uint16_t sc_h, uint16_t mn_h, const double* s, int flags,
                                double* out) {
  double sc = or_fp16_to_double(sc_h), mn = or_fp16_to_double(mn_h);
  for (int j = 0; j < OR_D; ++j) {
    int c = (codes[j / 4] >> (2 * (j % 4))) & 3;
    out[j] = mn + or_level(flags, c) * sc;
  }
  if (flags & OR_ROTATE) {
    or_wht128(out);
    for (int j = 0; j < OR_D; ++j) out[j] = s[j] * out[j] / (double)OR_D;
  }
}

/* Exported for the codec pins: r~ of one record (codes [32], fp16 scale and min). */
void or_dequantize_residual(const uint8_t* codes, uint16_t sc_h, uint16_t mn_h, uint64_t rot_seed, int flags,
                            double* out) {
  double s[OR_D];
  or_signs(rot_seed, s);
  or_dequant_residual(codes, sc_h, mn_h, s, flags, out);
}

/* x^_i of Eq. 3 for one side, for every position; out [S][128]. */
void or_reconstruct_side(int32_t S, const uint16_t* anchors, const uint16_t* idx, const uint16_t* gam, int32_t nres,
                         const int32_t* res, const uint8_t* codes, const uint16_t* scale, const uint16_t* mins,
                         uint64_t rot_seed, int flags, double* out) {
  double s[OR_D], rt[OR_D];
  or_signs(rot_seed, s);
  for (int32_t i = 0; i < S; ++i) {
    double g = or_fp16_to_double(gam[i]);
    const uint16_t* xa = anchors + (size_t)idx[i] * OR_D;
    for (int j = 0; j < OR_D; ++j) out[(size_t)i * OR_D + j] = g * or_bf16_to_double(xa[j]);
  }
  for (int32_t t = 0; t < nres; ++t) {
    or_dequant_residual(codes + (size_t)t * 32, scale[t], mins[t], s, flags, rt);
    for (int j = 0; j < OR_D; ++j) out[(size_t)res[t] * OR_D + j] += rt[j];
  }
}

/* RoPE (Section 3.2: keys kept pre-RoPE, the rotation applied at decode): the
 * rotate-half form, dimension pairs (j, j + 64) turned by the angle p theta_j
 * with theta_j = base^(-2j/128):
 *   y_j = x_j cos - x_{j+64} sin,   y_{j+64} = x_{j+64} cos + x_j sin. */
void or_rope(double* x, int64_t p, double base) {
  for (int j = 0; j < OR_D / 2; ++j) {
    double th = pow(base, -2.0 * (double)j / (double)OR_D);
    double a = (double)p * th;
    double c = cos(a), sn = sin(a);
    double x0 = x[j], x1 = x[j + OR_D / 2];
    x[j] = x0 * c - x1 * sn;
    x[j + OR_D / 2] = x1 * c + x0 * sn;
  }
}

/* Definitional attention for one unit with an exact dense suffix: G query
 * rows (bf16 bits [G][128]), out [G][128] fp64.  Each key and value of the
 * S compressed positions is rebuilt per Eq. 3; the nsuf suffix tokens (bf16
 * rows ksuf, vsuf [nsuf][128], kept exact: Appendix E.2) follow them, and the
 * softmax of Eq. 4 is taken over all S + nsuf positions at once (the combine
 * of Appendix E.1 attends both under the same softmax). */
void or_attend_unit_suffix(const or_unit* u, const uint16_t* q, int32_t G, double sm_scale, uint64_t rot_seed,
                           int flags, double rope_theta, const uint16_t* ksuf, const uint16_t* vsuf, int32_t nsuf,
                           double* out) {
  int32_t S = u->S;
  int32_t n = S + nsuf; /* positions of the softmax */
  double s[OR_D];
  or_signs(rot_seed, s);
  int32_t* slot_k = (int32_t*)malloc(sizeof(int32_t) * (size_t)S);
  int32_t* slot_v = (int32_t*)malloc(sizeof(int32_t) * (size_t)S);
  for (int32_t i = 0; i < S; ++i) slot_k[i] = slot_v[i] = -1;
  for (int32_t t = 0; t < u->nk; ++t) slot_k[u->res_k[t]] = t;
  for (int32_t t = 0; t < u->nv; ++t) slot_v[u->res_v[t]] = t;
  double* logit = (double*)malloc(sizeof(double) * (size_t)n * (size_t)G);
  double x[OR_D], rt[OR_D], qd[8][OR_D];
  for (int32_t g = 0; g < G; ++g)
    for (int j = 0; j < OR_D; ++j) qd[g][j] = or_bf16_to_double(q[(size_t)g * OR_D + j]);
  for (int32_t i = 0; i < n; ++i) {
    if (i < S) {
      double gk = or_fp16_to_double(u->gam_k[i]);
      const uint16_t* xa = u->anchor_k + (size_t)u->idx_k[i] * OR_D;
      for (int j = 0; j < OR_D; ++j) x[j] = gk * or_bf16_to_double(xa[j]);
      if (slot_k[i] >= 0) {
        int32_t t = slot_k[i];
        or_dequant_residual(u->codes_k + (size_t)t * 32, u->scale_k[t], u->min_k[t], s, flags, rt);
        for (int j = 0; j < OR_D; ++j) x[j] += rt[j];
      }
    } else {
      for (int j = 0; j < OR_D; ++j) x[j] = or_bf16_to_double(ksuf[(size_t)(i - S) * OR_D + j]);
    }
    if (flags & OR_ROPE) /* the key at its position: compressed i at pos[i], suffix t at S + t */
      or_rope(x, i < S ? (u->pos ? u->pos[i] : i) : i, rope_theta);
    for (int32_t g = 0; g < G; ++g) {
      double d = 0.0;
      for (int j = 0; j < OR_D; ++j) d += qd[g][j] * x[j];
      logit[(size_t)i * G + g] = sm_scale * d;
    }
  }
  for (int32_t g = 0; g < G; ++g) {
    double m = -INFINITY;
    for (int32_t i = 0; i < n; ++i)
      if (logit[(size_t)i * G + g] > m) m = logit[(size_t)i * G + g];
    double den = 0.0;
    for (int32_t i = 0; i < n; ++i) {
      double e = exp(logit[(size_t)i * G + g] - m);
      logit[(size_t)i * G + g] = e;
      den += e;
    }
    for (int32_t i = 0; i < n; ++i) logit[(size_t)i * G + g] /= den;
  }
  for (int32_t g = 0; g < G; ++g)
    for (int j = 0; j < OR_D; ++j) out[(size_t)g * OR_D + j] = 0.0;
  for (int32_t i = 0; i < n; ++i) {
    if (i < S) {
      double gv = or_fp16_to_double(u->gam_v[i]);
      const uint16_t* xa = u->anchor_v + (size_t)u->idx_v[i] * OR_D;
      for (int j = 0; j < OR_D; ++j) x[j] = gv * or_bf16_to_double(xa[j]);
      if (slot_v[i] >= 0) {
        int32_t t = slot_v[i];
        or_dequant_residual(u->codes_v + (size_t)t * 32, u->scale_v[t], u->min_v[t], s, flags, rt);
        for (int j = 0; j < OR_D; ++j) x[j] += rt[j];
      }
    } else {
      for (int j = 0; j < OR_D; ++j) x[j] = or_bf16_to_double(vsuf[(size_t)(i - S) * OR_D + j]);
    }
    for (int32_t g = 0; g < G; ++g) {
      double a = logit[(size_t)i * G + g];
      for (int j = 0; j < OR_D; ++j) out[(size_t)g * OR_D + j] += a * x[j];
    }
  }
  free(logit);
  free(slot_k);
  free(slot_v);
}

/* Definitional attention for one unit (no suffix): the softmax of Eq. 4 over
 * its S positions, each key and value rebuilt per Eq. 3. */
void or_attend_unit(const or_unit* u, const uint16_t* q, int32_t G, double sm_scale, uint64_t rot_seed, int flags,
                    double* out) {
  or_attend_unit_suffix(u, q, G, sm_scale, rot_seed, flags, 0.0, NULL, NULL, 0, out);
}

/* ------------------------------------------------------------------------ */
/* The paper's full selection (Algorithm 1): anchors scored by the          */
/* observation queries (Section 3.2, Appendix A.2), output-aware residual   */
/* utilities (Section 3.3, Eq. 6), the byte budget of Eq. 9 pooled over a   */
/* layer's KV heads (Section 3.4).                                           */
/* ------------------------------------------------------------------------ */

/* e^x for x <= 0 by the Cody-Waite argument reduction and a Taylor series
 * (Cody and Waite, "Software Manual for the Elementary Functions", 1980):
 * n = rint(x / ln 2), r = (x - n c1) - n c2 with c1 + c2 = ln 2 (c1 holding
 * the leading 32 bits, so n c1 is exact), then e^r = sum_{j<=22} r^j / j!
 * by Horner's rule, then the factor 2^n.  Every step is one separately
 * rounded IEEE operation in a fixed order, so any implementation of the same
 * steps gives the same bits; its error is about 1 ulp (pinned against libm).
 * Arguments below -700 give 0, so the scaling by 2^n never leaves the normal
 * range (there it is exact). */
double or_exp_neg(double x) {
  if (!(x >= -700.0)) return 0.0;
  const double c1 = 0.693147180559890330187045037746429443359375; /* 2^-32 grid */
  const double c2 = 5.4979230187083711552420206887987e-14;
  double n = rint(x / 0.6931471805599453094172321);
  double r = (x - n * c1) - n * c2;
  double y = 1.0;
  for (int j = 22; j >= 1; --j) y = 1.0 + (r / (double)j) * y;
  return ldexp(y, (int)n);
}

/* Exact attention of m query rows over the dense keys of one unit (Eq. 4,
 * logits q.K_t / sqrt(D), softmax over all S positions): alpha [m][S].
 * Sums run in position order. */
static void or_obs_alpha(int32_t S, int32_t m, const uint16_t* K, const uint16_t* Q, double* alpha) {
  const double inv = 1.0 / sqrt((double)OR_D);
  double qd[OR_D];
  for (int32_t w = 0; w < m; ++w) {
    for (int j = 0; j < OR_D; ++j) qd[j] = or_bf16_to_double(Q[(size_t)w * OR_D + j]);
    double* a = alpha + (size_t)w * S;
    double mx = -INFINITY;
    for (int32_t t = 0; t < S; ++t) {
      double d = 0.0;
      for (int j = 0; j < OR_D; ++j) d = d + qd[j] * or_bf16_to_double(K[(size_t)t * OR_D + j]);
      a[t] = d * inv;
      if (a[t] > mx) mx = a[t];
    }
    double den = 0.0;
    for (int32_t t = 0; t < S; ++t) {
      a[t] = or_exp_neg(a[t] - mx);
      den = den + a[t];
    }
    for (int32_t t = 0; t < S; ++t) a[t] = a[t] / den;
  }
}

/* Appendix A.2 selector score of the candidate positions t in [0, P), P = S - W:
 * the m observation rows' attention averaged over the rows, then average
 * pooling of odd width kappa centred on t, zero outside [0, P), divided by kappa. */
void or_selector_scores(int32_t S, int32_t P, int32_t m, int32_t kappa, const double* alpha, double* score) {
  double* mean = (double*)malloc(sizeof(double) * (size_t)(P > 0 ? P : 1));
  for (int32_t t = 0; t < P; ++t) {
    double acc = 0.0;
    for (int32_t w = 0; w < m; ++w) acc = acc + alpha[(size_t)w * S + t];
    mean[t] = acc / (double)m;
  }
  int32_t h = kappa / 2;
  for (int32_t t = 0; t < P; ++t) {
    double acc = 0.0;
    for (int32_t j = t - h; j <= t + h; ++j)
      if (j >= 0 && j < P) acc = acc + mean[j];
    score[t] = acc / (double)kappa;
  }
  free(mean);
}

/* Exported for the pins: the selector scores of one unit from its keys and m observation rows. */
void or_selector_scores_unit(int32_t S, int32_t W, int32_t m, int32_t kappa, const uint16_t* K, const uint16_t* Q,
                             double* score) {
  double* alpha = (double*)malloc(sizeof(double) * (size_t)m * (size_t)S + 1);
  or_obs_alpha(S, m, K, Q, alpha);
  int32_t w = W < S ? W : S;
  or_selector_scores(S, S - w, m, kappa, alpha, score);
  free(alpha);
}

typedef struct {
  double u;
  int32_t h, pos;
} or_util;

/* higher utility first; equal utilities: lower head, then lower position */
static int cmp_util_desc(const void* a, const void* b) {
  const or_util* x = (const or_util*)a;
  const or_util* y = (const or_util*)b;
  if (x->u > y->u) return -1;
  if (x->u < y->u) return 1;
  if (x->h != y->h) return (x->h < y->h) ? -1 : 1;
  return (x->pos < y->pos) ? -1 : (x->pos > y->pos);
}

/* Eq. 11 fixed bytes M_base and Eq. 9 residual count N of one layer of H KV
 * heads at context S (Appendix A.1 accounting: b_a = b_gamma = 2, residual
 * cost b_res = (c_K + c_V) / 2 with c_K = D/4 + 4 and c_V = D/4 + 5). */
int64_t or_budget_n(double theta, int32_t S, int32_t H, int32_t W, int32_t k) {
  int32_t w = W < S ? W : S;
  int64_t P = (int64_t)S - w;
  int64_t words = (P + 63) / 64;
  double m_full = 4.0 * (double)S * (double)H * (double)OR_D;
  double m_base = (double)H * (4.0 * k * OR_D + 8.0 * (k - w) + 2.0 * (double)P * (2 + 2)) + 24.0 * H * words +
                  8.0 * (H + 1) + 4.0 * (double)P;
  double b_res = ((OR_D / 4 + 4) + (OR_D / 4 + 5)) / 2.0;
  double n = floor((theta * m_full - m_base) / b_res);
  return n > 0.0 ? (int64_t)n : 0;
}

/*
 * Algorithm 1, per KV head: anchor set, assignment and coefficients, and the
 * Eq. 6 utilities of its non-anchor positions.  K, V bf16 [S][128] (rows of
 * one head, stride s_max), Q its m observation rows; u arrives with S and k
 * set.  cand[side] receive one entry per non-anchor position (*ncand of them).
 */
static int or_select_head(const uint16_t* Kh, const uint16_t* Vh, const uint16_t* Qh, int32_t m, int32_t W, float rho,
                          int32_t kappa, int32_t b, int32_t h, uint64_t seed, const double* sv, int flags, or_unit* u,
                          or_util* cand_k, or_util* cand_v, int64_t* ncand) {
  int32_t S = u->S, k = u->k;
  int32_t w = W < S ? W : S;
  int32_t rest = k - w;
  int32_t n_s = (m > 0 && rest > 0) ? (int32_t)floor((double)rho * (double)rest) : 0;
  double* alpha = (double*)malloc(sizeof(double) * (size_t)(m > 0 ? m : 1) * (size_t)S);
  double* y = (double*)malloc(sizeof(double) * (size_t)(m > 0 ? m : 1) * OR_D);
  if (m > 0) or_obs_alpha(S, m, Kh, Qh, alpha);
  /* anchor set: last w, top n_s by the selector score, the rest by the sampling hash */
  char* is_anchor = (char*)calloc((size_t)S, 1);
  int32_t P = S - w;
  if (rest > 0) {
    if (n_s > 0) {
      double* score = (double*)malloc(sizeof(double) * (size_t)P);
      or_selector_scores(S, P, m, kappa, alpha, score);
      or_util* sc = (or_util*)malloc(sizeof(or_util) * (size_t)P);
      for (int32_t t = 0; t < P; ++t) {
        sc[t].u = score[t];
        sc[t].h = 0;
        sc[t].pos = t;
      }
      qsort(sc, (size_t)P, sizeof(or_util), cmp_util_desc);
      for (int32_t t = 0; t < n_s; ++t) is_anchor[sc[t].pos] = 1;
      free(sc);
      free(score);
    }
    or_keypos* kp = (or_keypos*)malloc(sizeof(or_keypos) * (size_t)P);
    uint64_t base = seed ^ ((uint64_t)b << 40) ^ ((uint64_t)h << 32);
    int32_t np = 0;
    for (int32_t p = 0; p < P; ++p) {
      if (is_anchor[p]) continue;
      kp[np].key = or_splitmix64(base ^ (uint64_t)p);
      kp[np].pos = p;
      ++np;
    }
    qsort(kp, (size_t)np, sizeof(or_keypos), cmp_key_asc);
    for (int32_t t = 0; t < rest - n_s; ++t) is_anchor[kp[t].pos] = 1;
    free(kp);
  }
  for (int32_t p = S - w; p < S; ++p) is_anchor[p] = 1;
  int32_t* slot_of = (int32_t*)malloc(sizeof(int32_t) * (size_t)S);
  int32_t t = 0;
  for (int32_t p = 0; p < S; ++p) {
    if (is_anchor[p]) {
      u->anchor_pos[t] = p;
      slot_of[p] = t++;
    } else {
      slot_of[p] = -1;
    }
  }
  free(is_anchor);
  if (t != k) {
    free(slot_of);
    free(y);
    free(alpha);
    return -1;
  }
  for (int32_t a = 0; a < k; ++a) {
    memcpy(u->anchor_k + (size_t)a * OR_D, Kh + (size_t)u->anchor_pos[a] * OR_D, OR_D * 2);
    memcpy(u->anchor_v + (size_t)a * OR_D, Vh + (size_t)u->anchor_pos[a] * OR_D, OR_D * 2);
  }
  /* assignment and coefficients (Eq. 1, Eq. 2), no residual slots yet */
  or_encode_side(S, k, 0, Kh, u->anchor_pos, slot_of, sv, flags, u->idx_k, u->gam_k, NULL, NULL, NULL, NULL);
  or_encode_side(S, k, 0, Vh, u->anchor_pos, slot_of, sv, flags, u->idx_v, u->gam_v, NULL, NULL, NULL, NULL);
  /* exact outputs y^(w) of the observation rows (Eq. 4) */
  for (int32_t ww = 0; ww < m; ++ww)
    for (int j = 0; j < OR_D; ++j) {
      double acc = 0.0;
      for (int32_t p = 0; p < S; ++p)
        acc = acc + alpha[(size_t)ww * S + p] * or_bf16_to_double(Vh[(size_t)p * OR_D + j]);
      y[(size_t)ww * OR_D + j] = acc;
    }
  /* Eq. 6 utilities of the non-anchor positions, per side */
  int64_t nc = 0;
  for (int32_t p = 0; p < S; ++p) {
    if (slot_of[p] >= 0) continue;
    double rk[OR_D], rv[OR_D], vt[OR_D];
    double gk = or_fp16_to_double(u->gam_k[p]), gv = or_fp16_to_double(u->gam_v[p]);
    const uint16_t* xk = Kh + (size_t)p * OR_D;
    const uint16_t* xv = Vh + (size_t)p * OR_D;
    const uint16_t* ak = u->anchor_k + (size_t)u->idx_k[p] * OR_D;
    const uint16_t* av = u->anchor_v + (size_t)u->idx_v[p] * OR_D;
    double ev = 0.0;
    for (int j = 0; j < OR_D; ++j) {
      rk[j] = or_bf16_to_double(xk[j]) - gk * or_bf16_to_double(ak[j]);
      rv[j] = or_bf16_to_double(xv[j]) - gv * or_bf16_to_double(av[j]);
      vt[j] = or_bf16_to_double(xv[j]);
      ev = ev + rv[j] * rv[j];
    }
    double uk = 0.0, uv = 0.0;
    for (int32_t ww = 0; ww < m; ++ww) {
      double a = alpha[(size_t)ww * S + p];
      double a2 = a * a;
      double d = 0.0, dv = 0.0;
      for (int j = 0; j < OR_D; ++j) {
        d = d + or_bf16_to_double(Qh[(size_t)ww * OR_D + j]) * rk[j];
        double c = vt[j] - y[(size_t)ww * OR_D + j];
        dv = dv + c * c;
      }
      uk = uk + a2 * (d * d / (double)OR_D) * dv;
      uv = uv + a2 * ev;
    }
    if (m > 0) {
      uk = uk / (double)m;
      uv = uv / (double)m;
    }
    cand_k[nc].u = uk;
    cand_k[nc].h = h;
    cand_k[nc].pos = p;
    cand_v[nc].u = uv;
    cand_v[nc].h = h;
    cand_v[nc].pos = p;
    ++nc;
  }
  *ncand = nc;
  free(slot_of);
  free(y);
  free(alpha);
  return 0;
}

/* Algorithm 1, per request: the Eq. 9 budget, keys floor(N / 2) and values the
 * rest, each side's top N pooled over the request's H heads (the candidates of
 * head h at cand + h S), then rotation and quantization of the chosen residuals. */
static void or_pool_request(const uint16_t* K, const uint16_t* V, int32_t s_max, int32_t H, int32_t W, float theta,
                            const double* sv, int flags, or_unit* units, or_util* cand[2], const int64_t* ncand) {
  int32_t S = units[0].S, k = units[0].k;
  int64_t N = or_budget_n((double)theta, S, H, W, k);
  int64_t nside[2] = {N / 2, N - N / 2};
  for (int side = 0; side < 2; ++side) {
    /* gather the heads' candidates, then rank them */
    int64_t tot = 0;
    for (int32_t h = 0; h < H; ++h) {
      memmove(cand[side] + tot, cand[side] + (size_t)h * S, sizeof(or_util) * (size_t)ncand[h]);
      tot += ncand[h];
    }
    if (nside[side] > tot) nside[side] = tot;
    qsort(cand[side], (size_t)tot, sizeof(or_util), cmp_util_desc);
    for (int32_t h = 0; h < H; ++h) {
      if (side == 0) units[h].nk = 0;
      else units[h].nv = 0;
    }
    for (int64_t i = 0; i < nside[side]; ++i) {
      or_unit* u = &units[cand[side][i].h];
      if (side == 0) u->res_k[u->nk++] = cand[side][i].pos;
      else u->res_v[u->nv++] = cand[side][i].pos;
    }
  }
  /* rotate and quantize the chosen residuals (Appendix A.1), positions ascending */
  for (int32_t h = 0; h < H; ++h) {
    or_unit* u = &units[h];
    const uint16_t* Kh = K + (size_t)h * s_max * OR_D;
    const uint16_t* Vh = V + (size_t)h * s_max * OR_D;
    if (u->nk > 0) qsort(u->res_k, (size_t)u->nk, sizeof(int32_t), cmp_i32);
    if (u->nv > 0) qsort(u->res_v, (size_t)u->nv, sizeof(int32_t), cmp_i32);
    for (int side = 0; side < 2; ++side) {
      int32_t n = side ? u->nv : u->nk;
      const int32_t* res = side ? u->res_v : u->res_k;
      const uint16_t* X = side ? Vh : Kh;
      const uint16_t* A = side ? u->anchor_v : u->anchor_k;
      const uint16_t* idx = side ? u->idx_v : u->idx_k;
      const uint16_t* gam = side ? u->gam_v : u->gam_k;
      for (int32_t i = 0; i < n; ++i) {
        double r[OR_D];
        int32_t p = res[i];
        double g = or_fp16_to_double(gam[p]);
        for (int j = 0; j < OR_D; ++j)
          r[j] = or_bf16_to_double(X[(size_t)p * OR_D + j]) - g * or_bf16_to_double(A[(size_t)idx[p] * OR_D + j]);
        if (side == 0) or_quantize(r, sv, flags, u->codes_k + (size_t)i * 32, &u->scale_k[i], &u->min_k[i]);
        else or_quantize(r, sv, flags, u->codes_v + (size_t)i * 32, &u->scale_v[i], &u->min_v[i]);
      }
    }
  }
}

/* Exported for the pins: Eq. 6 utilities of every position of one unit with
 * given anchors and coefficients (anchors get -1).  K, V bf16 [S][128],
 * Q bf16 [m][128]; uk, uv [S]. */
void or_utilities_unit(const or_unit* u, const uint16_t* K, const uint16_t* V, const uint16_t* Q, int32_t m,
                       double* uk, double* uv) {
  int32_t S = u->S;
  double* alpha = (double*)malloc(sizeof(double) * (size_t)(m > 0 ? m : 1) * (size_t)S);
  double* y = (double*)malloc(sizeof(double) * (size_t)(m > 0 ? m : 1) * OR_D);
  if (m > 0) or_obs_alpha(S, m, K, Q, alpha);
  for (int32_t ww = 0; ww < m; ++ww)
    for (int j = 0; j < OR_D; ++j) {
      double acc = 0.0;
      for (int32_t p = 0; p < S; ++p) acc = acc + alpha[(size_t)ww * S + p] * or_bf16_to_double(V[(size_t)p * OR_D + j]);
      y[(size_t)ww * OR_D + j] = acc;
    }
  char* is_anchor = (char*)calloc((size_t)S, 1);
  for (int32_t a = 0; a < u->k; ++a) is_anchor[u->anchor_pos[a]] = 1;
  for (int32_t p = 0; p < S; ++p) {
    if (is_anchor[p]) {
      uk[p] = uv[p] = -1.0;
      continue;
    }
    double rk[OR_D], ev = 0.0;
    double gk = or_fp16_to_double(u->gam_k[p]), gv = or_fp16_to_double(u->gam_v[p]);
    for (int j = 0; j < OR_D; ++j) {
      rk[j] = or_bf16_to_double(K[(size_t)p * OR_D + j]) - gk * or_bf16_to_double(u->anchor_k[(size_t)u->idx_k[p] * OR_D + j]);
      double rv = or_bf16_to_double(V[(size_t)p * OR_D + j]) - gv * or_bf16_to_double(u->anchor_v[(size_t)u->idx_v[p] * OR_D + j]);
      ev = ev + rv * rv;
    }
    double a_k = 0.0, a_v = 0.0;
    for (int32_t ww = 0; ww < m; ++ww) {
      double a = alpha[(size_t)ww * S + p];
      double d = 0.0, dv = 0.0;
      for (int j = 0; j < OR_D; ++j) {
        d = d + or_bf16_to_double(Q[(size_t)ww * OR_D + j]) * rk[j];
        double c = or_bf16_to_double(V[(size_t)p * OR_D + j]) - y[(size_t)ww * OR_D + j];
        dv = dv + c * c;
      }
      a_k = a_k + (a * a) * (d * d / (double)OR_D) * dv;
      a_v = a_v + (a * a) * ev;
    }
    uk[p] = m > 0 ? a_k / (double)m : 0.0;
    uv[p] = m > 0 ? a_v / (double)m : 0.0;
  }
  free(is_anchor);
  free(y);
  free(alpha);
}

/* Batched over requests: K, V [B][H][s_max][128], Q [B][H][m][128]; units [B*H]
 * with S and k set and residual arrays sized min(N_side, S - k).  The heads
 * run in parallel, then each request's pooling. */
int or_encode_select_batch(const uint16_t* K, const uint16_t* V, const uint16_t* Q, int32_t s_max, int32_t B, int32_t H,
                           int32_t m, int32_t W, float theta, float rho, int32_t kappa, uint64_t seed,
                           uint64_t rot_seed, int flags, or_unit* units) {
  double sv[OR_D];
  or_signs(rot_seed, sv);
  int32_t n = B * H;
  or_util** ck = (or_util**)malloc(sizeof(or_util*) * (size_t)B);
  or_util** cv = (or_util**)malloc(sizeof(or_util*) * (size_t)B);
  int64_t* ncand = (int64_t*)calloc((size_t)n, sizeof(int64_t));
  for (int32_t b = 0; b < B; ++b) {
    size_t S = (size_t)units[(size_t)b * H].S;
    ck[b] = (or_util*)malloc(sizeof(or_util) * (size_t)H * S + 1);
    cv[b] = (or_util*)malloc(sizeof(or_util) * (size_t)H * S + 1);
  }
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
  for (int32_t u = 0; u < n; ++u) {
    int32_t b = u / H, h = u % H;
    size_t off = (size_t)u * (size_t)s_max * OR_D;
    size_t S = (size_t)units[u].S;
    if (or_select_head(K + off, V + off, Q + (size_t)u * (size_t)m * OR_D, m, W, rho, kappa, b, h, seed, sv, flags,
                       &units[u], ck[b] + (size_t)h * S, cv[b] + (size_t)h * S, &ncand[u]) != 0)
      bad |= 1;
  }
  if (!bad) {
#pragma omp parallel for schedule(dynamic, 1)
    for (int32_t b = 0; b < B; ++b) {
      size_t off = (size_t)b * H * (size_t)s_max * OR_D;
      or_util* cand[2] = {ck[b], cv[b]};
      or_pool_request(K + off, V + off, s_max, H, W, theta, sv, flags, units + (size_t)b * H, cand,
                      ncand + (size_t)b * H);
    }
  }
  for (int32_t b = 0; b < B; ++b) {
    free(ck[b]);
    free(cv[b]);
  }
  free(ck);
  free(cv);
  free(ncand);
  return bad ? -1 : 0;
}

/* Batched definitional attention: q bf16 [n_units][G][128] (unit u = b*H + h
 * owns query heads h*G .. h*G+G-1 of request b), out fp64 same shape.
 * Units with sel[u] == 0 are skipped (sel may be NULL). */
void or_attend_batch(const or_unit* units, int32_t n_units, const uint16_t* q, int32_t G, double sm_scale,
                     uint64_t rot_seed, int flags, double rope_theta, const uint8_t* sel, double* out) {
#pragma omp parallel for schedule(dynamic, 1)
  for (int32_t u = 0; u < n_units; ++u) {
    if (sel && !sel[u]) continue;
    or_attend_unit_suffix(&units[u], q + (size_t)u * G * OR_D, G, sm_scale, rot_seed, flags, rope_theta, NULL, NULL, 0,
                          out + (size_t)u * G * OR_D);
  }
}

/* Batched attention with exact dense suffixes: unit u = b*H + h attends its
 * S positions and the first suf_len[b] rows of its suffix block, rows
 * ksuf/vsuf + (u * suf_cap + t) * 128 (bf16). */
void or_attend_batch_suffix(const or_unit* units, int32_t n_units, int32_t H, const uint16_t* q, int32_t G,
                            double sm_scale, uint64_t rot_seed, int flags, double rope_theta, const uint16_t* ksuf,
                            const uint16_t* vsuf, const int32_t* suf_len, int32_t suf_cap, double* out) {
#pragma omp parallel for schedule(dynamic, 1)
  for (int32_t u = 0; u < n_units; ++u) {
    const size_t base = (size_t)u * (size_t)suf_cap * OR_D;
    or_attend_unit_suffix(&units[u], q + (size_t)u * G * OR_D, G, sm_scale, rot_seed, flags, rope_theta, ksuf + base,
                          vsuf + base,
                          suf_len[u / H], out + (size_t)u * G * OR_D);
  }
}

/* The same attention regrouped by anchor: anchor scores once per anchor,
 * value weights summed per anchor before one product with the anchor values,
 * and the inverse rotation applied once to the accumulated residual codes. */
void or_attend_factorized(const or_unit* u, const uint16_t* q, int32_t G, double sm_scale, uint64_t rot_seed,
                          int flags, double* out) {
  int32_t S = u->S, k = u->k;
  double s[OR_D];
  or_signs(rot_seed, s);
  double qd[8][OR_D], qr[8][OR_D], qsum[8];
  for (int32_t g = 0; g < G; ++g) {
    for (int j = 0; j < OR_D; ++j) qd[g][j] = or_bf16_to_double(q[(size_t)g * OR_D + j]);
    for (int j = 0; j < OR_D; ++j) qr[g][j] = (flags & OR_ROTATE) ? s[j] * qd[g][j] : qd[g][j];
    if (flags & OR_ROTATE) {
      or_wht128(qr[g]);
      for (int j = 0; j < OR_D; ++j) qr[g][j] /= (double)OR_D;
    }
    qsum[g] = 0.0;
    for (int j = 0; j < OR_D; ++j) qsum[g] += qr[g][j];
  }
  double* sa = (double*)malloc(sizeof(double) * (size_t)(k ? k : 1) * G);
  for (int32_t a = 0; a < k; ++a)
    for (int32_t g = 0; g < G; ++g) {
      double d = 0.0;
      for (int j = 0; j < OR_D; ++j) d += qd[g][j] * or_bf16_to_double(u->anchor_k[(size_t)a * OR_D + j]);
      sa[(size_t)a * G + g] = d;
    }
  double* lg = (double*)malloc(sizeof(double) * (size_t)S * G);
  for (int32_t i = 0; i < S; ++i)
    for (int32_t g = 0; g < G; ++g)
      lg[(size_t)i * G + g] = or_fp16_to_double(u->gam_k[i]) * sa[(size_t)u->idx_k[i] * G + g];
  for (int32_t t = 0; t < u->nk; ++t) {
    int32_t i = u->res_k[t];
    double sc = or_fp16_to_double(u->scale_k[t]), mn = or_fp16_to_double(u->min_k[t]);
    for (int32_t g = 0; g < G; ++g) {
      double d = 0.0;
      for (int j = 0; j < OR_D; ++j)
        d += qr[g][j] * or_level(flags, (u->codes_k[(size_t)t * 32 + j / 4] >> (2 * (j % 4))) & 3);
      lg[(size_t)i * G + g] += mn * qsum[g] + sc * d;
    }
  }
  for (int32_t g = 0; g < G; ++g) {
    double m = -INFINITY, den = 0.0;
    for (int32_t i = 0; i < S; ++i) {
      lg[(size_t)i * G + g] *= sm_scale;
      if (lg[(size_t)i * G + g] > m) m = lg[(size_t)i * G + g];
    }
    for (int32_t i = 0; i < S; ++i) {
      lg[(size_t)i * G + g] = exp(lg[(size_t)i * G + g] - m);
      den += lg[(size_t)i * G + g];
    }
    for (int32_t i = 0; i < S; ++i) lg[(size_t)i * G + g] /= den;
  }
  double* w = (double*)calloc((size_t)(k ? k : 1) * G, sizeof(double));
  for (int32_t i = 0; i < S; ++i)
    for (int32_t g = 0; g < G; ++g)
      w[(size_t)u->idx_v[i] * G + g] += lg[(size_t)i * G + g] * or_fp16_to_double(u->gam_v[i]);
  double acc[8][OR_D];
  for (int32_t g = 0; g < G; ++g)
    for (int j = 0; j < OR_D; ++j) acc[g][j] = 0.0;
  for (int32_t t = 0; t < u->nv; ++t) {
    int32_t i = u->res_v[t];
    double sc = or_fp16_to_double(u->scale_v[t]), mn = or_fp16_to_double(u->min_v[t]);
    for (int32_t g = 0; g < G; ++g) {
      double p = lg[(size_t)i * G + g];
      for (int j = 0; j < OR_D; ++j)
        acc[g][j] += p * (mn + sc * or_level(flags, (u->codes_v[(size_t)t * 32 + j / 4] >> (2 * (j % 4))) & 3));
    }
  }
  for (int32_t g = 0; g < G; ++g) {
    if (flags & OR_ROTATE) {
      or_wht128(acc[g]);
      for (int j = 0; j < OR_D; ++j) acc[g][j] = s[j] * acc[g][j] / (double)OR_D;
    }
    for (int j = 0; j < OR_D; ++j) {
      double o = acc[g][j];
      for (int32_t a = 0; a < k; ++a) o += w[(size_t)a * G + g] * or_bf16_to_double(u->anchor_v[(size_t)a * OR_D + j]);
      out[(size_t)g * OR_D + j] = o;
    }
  }
  free(w);
  free(lg);
  free(sa);
}

/* ------------------------------------------------------------------------ */
/* Independent reader of the packed arena                                    */
/* ------------------------------------------------------------------------ */

/* Header: magic u32 @0, version u32 @4, total_bytes u64 @8, params (56 B) @16,
 * n_units i32 @72, max_len i32 @76, desc_offset u64 @80, sign bits 2 x u64 @88.
 * Descriptor (256 B each at desc_offset + 256 u): len, k, n_res_k, n_res_v,
 * n_tiles, b, h, reserved (i32 each), then u64: offsets of anchor_k, anchor_v,
 * anchor_pos, tile table, tile blocks; tiles capacity, data_bytes, and the
 * offset of the positions (RoPE arenas). */
static uint32_t rd32(const uint8_t* p) {
  uint32_t v;
  memcpy(&v, p, 4);
  return v;
}
static uint64_t rd64(const uint8_t* p) {
  uint64_t v;
  memcpy(&v, p, 8);
  return v;
}

/* Returns 0 and the shape of unit u, or -1 on a malformed arena. */
int or_arena_shape(const uint8_t* arena, uint64_t bytes, int32_t u, int32_t* shape4) {
  if (bytes < 256 || rd32(arena) != 0x32564B41u || rd32(arena + 4) != 4u || rd32(arena + 104) != 1024u) return -1;
  int32_t n_units = (int32_t)rd32(arena + 72);
  uint64_t doff = rd64(arena + 80);
  if (u < 0 || u >= n_units || doff + 256ull * (uint64_t)(u + 1) > bytes) return -1;
  const uint8_t* d = arena + doff + 256ull * (uint64_t)u;
  for (int t = 0; t < 4; ++t) shape4[t] = (int32_t)rd32(d + 4 * t);
  return 0;
}

/* Copies unit u's logical arrays out of the arena (shape first from
 * or_arena_shape).  The arena keeps tokens in its stored order (sorted by value
 * anchor slot); the arrays come back in that order, and res_k / res_v hold the
 * stored indices of the tokens with a residual.  Returns 0, or -1 on any
 * inconsistency (tile table, rank words, record counts, anchor slot range,
 * value slots out of order). */
int or_arena_unpack(const uint8_t* arena, uint64_t bytes, int32_t u, or_unit* out) {
  int32_t sh[4];
  if (or_arena_shape(arena, bytes, u, sh) != 0) return -1;
  const uint8_t* d = arena + rd64(arena + 80) + 256ull * (uint64_t)u;
  int32_t S = sh[0], k = sh[1], nk = sh[2], nv = sh[3];
  const int32_t T = 1024;
  int32_t nt = (int32_t)rd32(d + 16);
  if (nt != (S + T - 1) / T) return -1;
  uint64_t o_ak = rd64(d + 32), o_av = rd64(d + 40), o_ap = rd64(d + 48), o_tt = rd64(d + 56), o_ti = rd64(d + 64);
  uint64_t cap = rd64(d + 72);
  if (o_ak + 256ull * k > bytes || o_av + 256ull * k > bytes || o_ap + 4ull * k > bytes ||
      o_tt + 4ull * (2 * nt + 1) > bytes || o_ti + cap > bytes || (o_ak % 16) || (o_av % 16) || (o_ti % 16))
    return -1;
  for (int32_t a = 0; a < k; ++a)
    for (int c = 0; c < 16; ++c) {
      memcpy(out->anchor_k + (size_t)a * 128 + 8 * c, arena + o_ak + (size_t)a * 256 + 16 * (c ^ (a & 7)), 16);
      memcpy(out->anchor_v + (size_t)a * 128 + 8 * c, arena + o_av + (size_t)a * 256 + 16 * (c ^ (a & 7)), 16);
    }
  memcpy(out->anchor_pos, arena + o_ap, (size_t)k * 4);
  int32_t cnt[2] = {0, 0};
  uint32_t prev_av = 0;
  for (int32_t j = 0; j < nt; ++j) {
    uint32_t b0 = rd32(arena + o_tt + 4ull * j), b1 = rd32(arena + o_tt + 4ull * (j + 1));
    if ((b0 % 16) || b1 < b0 || b1 > cap) return -1;
    const uint8_t* blk = arena + o_ti + b0;
    int32_t n = S - j * T < T ? S - j * T : T;
    int32_t nw = (n + 63) / 64, n64 = 64 * nw;
    const uint8_t* kst = blk;
    const uint8_t* vst = blk + 4ull * n64;
    const uint8_t* bm[2] = {blk + 8ull * n64, blk + 8ull * n64 + 8ull * nw};
    int32_t rk_pad = ((2 * nw + 15) / 16) * 16;
    const uint8_t* rk[2] = {blk + 8ull * n64 + 16ull * nw, blk + 8ull * n64 + 16ull * nw + rk_pad};
    uint32_t F = 8u * n64 + 16u * nw + 2u * rk_pad;
    /* records of this tile, per side */
    int32_t m[2] = {0, 0};
    for (int side = 0; side < 2; ++side)
      for (int32_t w = 0; w < nw; ++w) {
        uint64_t word = rd64(bm[side] + 8ull * w);
        if ((uint32_t)(rd32(rk[side] + 2ull * w) & 0xFFFFu) != (uint32_t)m[side]) return -1;
        if (w == nw - 1 && n % 64 && (word >> (n % 64))) return -1; /* bits past the last token */
        for (int bit = 0; bit < 64; ++bit) m[side] += (int32_t)((word >> bit) & 1ull);
      }
    uint32_t sm_off[2] = {F, F + (uint32_t)(((4 * m[0] + 15) / 16) * 16)};
    uint32_t cd_off[2];
    cd_off[0] = sm_off[1] + (uint32_t)(((4 * m[1] + 15) / 16) * 16);
    cd_off[1] = cd_off[0] + 32u * (uint32_t)m[0];
    /* value codes: groups of 16 records, dimension-major (word 32 (d/32) + 4 (d%8) + (d%32)/8
     * of a group holds dimension d, record slot s at bits 2 (s/2) + 16 (s%2)) */
    uint32_t nvgrp = (uint32_t)((m[1] + 15) / 16);
    if (b0 + cd_off[1] + 512u * nvgrp != b1) return -1;
    for (int32_t sl = m[1]; sl < 16 * (int32_t)nvgrp; ++sl) /* padding slots hold zero codes */
      for (int dd = 0; dd < 128; ++dd) {
        uint32_t wd = rd32(blk + cd_off[1] + 512u * (uint32_t)(sl / 16) +
                           4u * (uint32_t)(32 * (dd / 32) + 4 * (dd % 8) + (dd % 32) / 8));
        if ((wd >> (2 * ((sl % 16) / 2) + 16 * (sl % 2))) & 3u) return -1;
      }
    if (cnt[0] + m[0] > nk || cnt[1] + m[1] > nv) return -1;
    int32_t r[2] = {0, 0};
    for (int32_t t = 0; t < n; ++t) {
      int32_t i = j * T + t;
      uint32_t ek = rd32(kst + 4ull * t), ev = rd32(vst + 4ull * t);
      out->idx_k[i] = (uint16_t)(ek & 0xFFFFu);
      out->gam_k[i] = (uint16_t)(ek >> 16);
      out->idx_v[i] = (uint16_t)(ev & 0xFFFFu);
      out->gam_v[i] = (uint16_t)(ev >> 16);
      if (out->idx_k[i] >= k || out->idx_v[i] >= k || (ev & 0xFFFFu) < prev_av) return -1;
      prev_av = ev & 0xFFFFu;
      for (int side = 0; side < 2; ++side) {
        if (!((rd64(bm[side] + 8ull * (t >> 6)) >> (t & 63)) & 1ull)) continue;
        int32_t g = cnt[side] + r[side];
        (side ? out->res_v : out->res_k)[g] = i;
        uint32_t e = rd32(blk + sm_off[side] + 4ull * r[side]);
        (side ? out->scale_v : out->scale_k)[g] = (uint16_t)(e & 0xFFFFu);
        (side ? out->min_v : out->min_k)[g] = (uint16_t)(e >> 16);
        if (side == 0) {
          memcpy(out->codes_k + 32ull * g, blk + cd_off[0] + 32ull * r[0], 32);
        } else {
          uint8_t* rec = out->codes_v + 32ull * g;
          memset(rec, 0, 32);
          for (int dd = 0; dd < 128; ++dd) {
            uint32_t wd = rd32(blk + cd_off[1] + 512u * (uint32_t)(r[1] / 16) +
                               4u * (uint32_t)(32 * (dd / 32) + 4 * (dd % 8) + (dd % 32) / 8));
            rec[dd / 4] |= (uint8_t)(((wd >> (2 * ((r[1] % 16) / 2) + 16 * (r[1] % 2))) & 3u) << (2 * (dd % 4)));
          }
        }
        ++r[side];
      }
    }
    for (int32_t t = n; t < n64; ++t)
      if (rd32(kst + 4ull * t) || rd32(vst + 4ull * t)) return -1;
    /* the tile's value-slot range word: slots of its first and last stored tokens */
    if (rd32(arena + o_tt + 4ull * (nt + 1 + j)) != ((rd32(vst) & 0xFFFFu) | ((rd32(vst + 4ull * (n - 1)) & 0xFFFFu) << 16)))
      return -1;
    cnt[0] += m[0];
    cnt[1] += m[1];
  }
  if (cnt[0] != nk || cnt[1] != nv) return -1;
  /* RoPE arenas (flags @64 of the header) keep each stored token's original position: a
   * permutation of 0 .. S-1, ascending among the tokens of one value slot (the stable sort) */
  if (rd32(arena + 64) & OR_ROPE) {
    uint64_t o_pos = rd64(d + 88);
    if (o_pos == 0 || o_pos + 4ull * S > bytes) return -1;
    uint8_t* seen = (uint8_t*)calloc((size_t)S, 1);
    int bad = 0;
    for (int32_t i = 0; i < S && !bad; ++i) {
      uint32_t p = rd32(arena + o_pos + 4ull * i);
      if (p >= (uint32_t)S || seen[p]) bad = 1;
      else seen[p] = 1;
      if (!bad && i > 0 && out->idx_v[i] == out->idx_v[i - 1] && p <= rd32(arena + o_pos + 4ull * (i - 1))) bad = 1;
      if (!bad && out->pos) out->pos[i] = (int32_t)p;
    }
    free(seen);
    if (bad) return -1;
  } else if (out->pos) {
    for (int32_t i = 0; i < S; ++i) out->pos[i] = -1; /* positions are not stored */
  }
  return 0;
}
