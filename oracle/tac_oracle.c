/*
 * TurboAngle CPU oracle (arXiv 2603.27467) -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, fp64 restatement of what the paper's encode/decode path
 * computes, written to check the CUDA path against.  It uses a DENSE
 * normalized Sylvester-Hadamard matrix (O(d^2) per vector), not a butterfly,
 * and shares no code, header, table or constant with the product library.
 * Only tests/, __graft_entry__.smoke() and bench.py (its CPU-baseline and
 * reference legs) may load or call it; the product path never does.
 *
 * Paper passages followed (section / equation / algorithm of the paper):
 *   - normalized Hadamard H, H = H^T = H^-1, norm preserving ......... Sec. 2
 *   - random +-1 diagonal D, y = H D x ................................ Sec. 2, Alg. 1
 *   - pair polar form r_i, theta_i = atan2(y_{2i+1}, y_{2i}) ........... Alg. 1
 *   - k_i = round(n theta_i / 2 pi) mod n ............................. Alg. 1
 *   - reconstruction y^_{2i} = r cos(2 pi k / n), x^ = D H y^ ......... Sec. 3.1
 *   - per-vector min-max norm quantization, fp32 min/max .............. Sec. 3.3, Eq. 2
 *   - log-space variant (Eq. 2 applied to log r) ...................... Sec. 3.3
 *   - average angle rate .............................................. Sec. 3.2, Eq. 1
 *   - total rate b_angle + b_norm/2 + 64/d ............................ Sec. 3.3, Eq. 3
 *
 * Readings of points the paper leaves open (each is also listed in the
 * design notes):
 *   R1 Hadamard order: Sylvester (natural) order, H[a][j] = (-1)^popcount(a&j)/sqrt(d).
 *   R2 Rounding in Alg. 1: k = floor(n theta/(2 pi) + 1/2) mod n, theta in (-pi, pi]
 *      from atan2; a value exactly halfway rounds up.
 *   R3 A pair (0, 0) gets k = 0.
 *   R4 Eq. 2 takes r_min and r_max as what the formula names: the minimum and the
 *      maximum of the vector's pair norms themselves (their fp64 values here).  Sec. 3.3
 *      stores the two in fp32 for the decoder: the header holds (float)r_min and
 *      (float)r_max (round to nearest), and decode dequantizes against those stored
 *      values.  Eq. 2's value is rounded half up and clamped to [0, 2^b - 1].
 *   R5 If r_max equals r_min every norm code is 0; if the stored r_max equals the
 *      stored r_min, decode returns the stored r_min for every pair (an all-zero vector
 *      decodes to zero).
 *   R6 Log-space: norms are floored at 2^-24 * r_max before the logarithm (so a zero
 *      pair norm has a finite code) and the stored r_min is that floored minimum;
 *      log base 2.
 *   R7 Dequantization (the paper states only the encode side): linear
 *      r^ = r_min + c (r_max - r_min)/(2^b - 1); log r^ = 2^(l_min + c (l_max - l_min)/(2^b - 1)).
 *   R8 Signs D: s_j = -1 iff bit 63 of SplitMix64 output #j of the stream seeded with
 *      key = SplitMix64 output #q of the stream seeded with `seed`, q = 2*layer + kv
 *      (q = 0 for every (layer, kv) in "shared" mode, the paper's single D).
 *   R9 Bit packing: each vector's codes form one LSB-first bitstream (code in slot
 *      v at bit v*w); a vector's stream starts on a byte boundary.  Slot v holds
 *      the code of pair phi_d(v) (orc_slot_pair: the natural order for d <= 32, a
 *      fixed relabeling of the pair-index bits for d = 64, 128).
 *   R16 fp32 norm storage (mode 2, the angle-only configuration whose rates count
 *      angle bits only, Sec. 3.1 and Tables 1-4): each pair norm r_i is stored as
 *      the fp32 value nearest to it (its 32 bits are the "norm code", b = 32) and
 *      decode uses that value as r^; there is no min/max header in this mode.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_TWO_PI (2.0 * 3.14159265358979323846)

/* ------------------------------------------------------------------------ */
/* SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom number     */
/* generators", OOPSLA 2014): state += 0x9E3779B97F4A7C15, then the         */
/* variant-13 finalizer.  Output #i (0-based) of the stream seeded with s is */
/* finalize(s + (i+1) * golden).  Used for the sign vector D (reading R8).  */
/* ------------------------------------------------------------------------ */
uint64_t orc_splitmix64(uint64_t seed, uint64_t i) {
  uint64_t z = seed + (i + 1u) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

/* Random +-1 diagonal D of Sec. 2 ("s_i ~ Uniform{+1,-1}"), one per (layer, K/V),
 * or one shared D as in the paper's implementation note (Sec. 3.1). */
void orc_signs(uint64_t seed, int layer, int kv, int shared, int d, int8_t* s) {
  uint64_t q = shared ? 0u : (uint64_t)(2 * layer + kv);
  uint64_t key = orc_splitmix64(seed, q);
  for (int j = 0; j < d; ++j) s[j] = (orc_splitmix64(key, (uint64_t)j) >> 63) ? -1 : 1;
}

static int popcount_u32(uint32_t v) {
  int c = 0;
  while (v) { c += (int)(v & 1u); v >>= 1; }
  return c;
}

/* Normalized Hadamard matrix of Sec. 2, Sylvester order (reading R1):
 * H[a][j] = (-1)^popcount(a & j) / sqrt(d), row-major d x d. */
void orc_hadamard(int d, double* H) {
  double scale = 1.0 / sqrt((double)d);
  for (int a = 0; a < d; ++a)
    for (int j = 0; j < d; ++j)
      H[(size_t)a * d + j] = (popcount_u32((uint32_t)(a & j)) & 1) ? -scale : scale;
}

/* y = H D x for one vector (Alg. 1, first step), dense matrix-vector product.
 * H = (1/sqrt d) * (+-1 matrix) (Sec. 2): the +-1 sum is formed first and scaled
 * once, so a coordinate that is exactly zero stays exactly zero (reading R3 then
 * applies to exactly the pairs that are (0, 0)). */
static void transform_one(const double* H, int d, const int8_t* s, const double* x, double* y) {
  const double scale = 1.0 / sqrt((double)d);
  for (int a = 0; a < d; ++a) {
    double acc = 0.0;
    for (int j = 0; j < d; ++j) {
      const double t = (double)s[j] * x[j];
      acc += (H[(size_t)a * d + j] < 0.0) ? -t : t;
    }
    y[a] = acc * scale;
  }
}

/* Public form of the transform for tests: rows x d in, rows x d out. */
int orc_transform(const double* x, int64_t rows, int d, const int8_t* s, double* y) {
  if (d <= 0 || (d & (d - 1))) return 1;
  double* H = (double*)malloc(sizeof(double) * (size_t)d * d);
  if (!H) return 2;
  orc_hadamard(d, H);
  for (int64_t r = 0; r < rows; ++r) transform_one(H, d, s, x + r * d, y + r * d);
  free(H);
  return 0;
}

/* Alg. 1: theta -> k.  Returns k in [0, n); writes the distance of theta to
 * the nearest bin edge ((k + 1/2) 2 pi / n), in radians, to *edge_dist. */
static int32_t angle_code(double y0, double y1, int n, double* edge_dist) {
  if (y0 == 0.0 && y1 == 0.0) {          /* reading R3 */
    *edge_dist = M_PI / n;               /* a zero pair sits on a bin centre */
    return 0;
  }
  double theta = atan2(y1, y0);           /* (-pi, pi] */
  double v = (double)n * theta / ORC_TWO_PI;
  double f = floor(v + 0.5);              /* reading R2 */
  *edge_dist = fabs(v - (floor(v) + 0.5)) * ORC_TWO_PI / n;
  long long k = (long long)f % n;
  if (k < 0) k += n;
  return (int32_t)k;
}

/* fp32 bit pattern of the float nearest to v (reading R16). */
static int32_t fp32_bits(double v) {
  float f = (float)v;
  int32_t b;
  memcpy(&b, &f, sizeof b);
  return b;
}

/* Eq. 2 with clamp (readings R4, R5); returns the pre-round value in *pre. */
static int32_t norm_code(double val, double lo, double hi, int b, double* pre) {
  int32_t L = (1 << b) - 1;
  if (hi == lo) { *pre = 0.0; return 0; }           /* reading R5 */
  double v = (val - lo) / (hi - lo) * (double)L;
  *pre = v;
  double c = floor(v + 0.5);
  if (c < 0.0) c = 0.0;
  if (c > (double)L) c = (double)L;
  return (int32_t)c;
}

/*
 * Encode (Alg. 1 + Sec. 3.3 / Eq. 2).
 *   x        rows x d doubles (the input vectors, converted exactly from bf16/fp32)
 *   s        d signs (+-1), the diagonal D
 *   n        angle bins; b norm bits; mode 0 = linear, 1 = log-space,
 *            2 = fp32 norms (b = 32, reading R16)
 *   k_out    rows x d/2 angle indices
 *   c_out    rows x d/2 norm codes
 *   hdr_out  rows x 2 floats: stored (r_min, r_max)
 *   edge_out rows x d/2 distances of theta_i to its nearest bin edge, radians (nullable)
 *   pre_out  rows x d/2 pre-round Eq. 2 values, in code units (nullable)
 *   r_out    rows x d/2 exact pair norms r_i (nullable)
 */
int orc_encode(const double* x, int64_t rows, int d, const int8_t* s, int n, int b, int mode,
               int32_t* k_out, int32_t* c_out, float* hdr_out, double* edge_out, double* pre_out,
               double* r_out) {
  if (d < 2 || (d & (d - 1)) || n < 1) return 1;
  if (!((mode == 0 || mode == 1) && b >= 1 && b <= 16) && !(mode == 2 && b == 32)) return 1;
  const int P = d / 2;
  double* H = (double*)malloc(sizeof(double) * (size_t)d * d);
  double* y = (double*)malloc(sizeof(double) * (size_t)d);
  double* r = (double*)malloc(sizeof(double) * (size_t)P);
  if (!H || !y || !r) { free(H); free(y); free(r); return 2; }
  orc_hadamard(d, H);
  for (int64_t row = 0; row < rows; ++row) {
    transform_one(H, d, s, x + row * d, y);
    double rmin = INFINITY, rmax = 0.0;
    for (int i = 0; i < P; ++i) {
      double y0 = y[2 * i], y1 = y[2 * i + 1];
      r[i] = sqrt(y0 * y0 + y1 * y1);                      /* Alg. 1 */
      double ed;
      k_out[row * P + i] = angle_code(y0, y1, n, &ed);     /* Alg. 1 */
      if (edge_out) edge_out[row * P + i] = ed;
      if (r_out) r_out[row * P + i] = r[i];
      if (r[i] < rmin) rmin = r[i];
      if (r[i] > rmax) rmax = r[i];
    }
    double* pre = pre_out ? pre_out + row * P : NULL;
    if (mode == 2) {                                         /* reading R16 */
      hdr_out[2 * row] = (float)rmin;
      hdr_out[2 * row + 1] = (float)rmax;
      for (int i = 0; i < P; ++i) {
        c_out[row * P + i] = fp32_bits(r[i]);
        if (pre) pre[i] = 0.0;
      }
    } else if (mode == 0) {
      hdr_out[2 * row] = (float)rmin;                         /* Sec. 3.3: stored in fp32 */
      hdr_out[2 * row + 1] = (float)rmax;
      for (int i = 0; i < P; ++i) {
        double pv;
        c_out[row * P + i] = norm_code(r[i], rmin, rmax, b, &pv);   /* Eq. 2, reading R4 */
        if (pre) pre[i] = pv;
      }
    } else {
      double floor_r = ldexp(rmax, -24);                     /* reading R6 */
      double lo = rmin < floor_r ? floor_r : rmin;
      hdr_out[2 * row] = (float)lo;                           /* Sec. 3.3: stored in fp32 */
      hdr_out[2 * row + 1] = (float)rmax;
      double lmin = (lo > 0.0) ? log2(lo) : 0.0;
      double lmax = (rmax > 0.0) ? log2(rmax) : 0.0;
      for (int i = 0; i < P; ++i) {
        double pv;
        if (rmax == lo) {                                     /* reading R5 */
          c_out[row * P + i] = 0;
          pv = 0.0;
        } else {
          double ri = r[i] < floor_r ? floor_r : r[i];
          c_out[row * P + i] = norm_code(log2(ri), lmin, lmax, b, &pv);  /* Sec. 3.3 log-space */
        }
        if (pre) pre[i] = pv;
      }
    }
  }
  free(H); free(y); free(r);
  return 0;
}

/*
 * Decode (Sec. 3.1 reconstruction + reading R7): r^ from the norm code and the
 * stored header, y^ = r^ (cos, sin)(2 pi k / n), x^ = D H y^ (dense).
 *   y_out rows x d doubles.
 */
int orc_decode(const int32_t* k, const int32_t* c, const float* hdr, int64_t rows, int d,
               const int8_t* s, int n, int b, int mode, double* y_out) {
  if (d < 2 || (d & (d - 1)) || n < 1) return 1;
  if (!((mode == 0 || mode == 1) && b >= 1 && b <= 16) && !(mode == 2 && b == 32)) return 1;
  const int P = d / 2;
  const double L = mode == 2 ? 1.0 : (double)((1 << b) - 1);
  double* H = (double*)malloc(sizeof(double) * (size_t)d * d);
  double* yh = (double*)malloc(sizeof(double) * (size_t)d);
  if (!H || !yh) { free(H); free(yh); return 2; }
  orc_hadamard(d, H);
  for (int64_t row = 0; row < rows; ++row) {
    double hmin = (double)hdr[2 * row], hmax = (double)hdr[2 * row + 1];
    for (int i = 0; i < P; ++i) {
      double ci = (double)c[row * P + i], rh;
      if (mode == 2) {                                       /* reading R16 */
        float f;
        memcpy(&f, &c[row * P + i], sizeof f);
        rh = (double)f;
      } else if (hmax == hmin) rh = hmin;
      else if (mode == 0) rh = hmin + ci * (hmax - hmin) / L;
      else {
        double lmin = log2(hmin), lmax = log2(hmax);
        rh = exp2(lmin + ci * (lmax - lmin) / L);
      }
      double phi = ORC_TWO_PI * (double)k[row * P + i] / (double)n;
      yh[2 * i] = rh * cos(phi);
      yh[2 * i + 1] = rh * sin(phi);
    }
    /* x^ = D H y^ : H is symmetric (Sec. 2), so row a of H is column a; the
     * +-1 sum is formed first and scaled by 1/sqrt(d) once. */
    double* out = y_out + row * d;
    const double scale = 1.0 / sqrt((double)d);
    for (int j = 0; j < d; ++j) {
      double acc = 0.0;
      for (int a = 0; a < d; ++a) acc += (H[(size_t)j * d + a] < 0.0) ? -yh[a] : yh[a];
      out[j] = (double)s[j] * (acc * scale);
    }
  }
  free(H); free(yh);
  return 0;
}

/* Reading R9: pack `count` codes of `bits` bits per row into an LSB-first
 * bitstream; row stride = ceil(count*bits/8) bytes. */
int orc_pack(const int32_t* codes, int64_t rows, int count, int bits, uint8_t* out) {
  if (bits < 1 || bits > 32) return 1;
  size_t stride = ((size_t)count * bits + 7) / 8;
  memset(out, 0, stride * (size_t)rows);
  for (int64_t r = 0; r < rows; ++r) {
    uint8_t* o = out + (size_t)r * stride;
    for (int i = 0; i < count; ++i) {
      uint32_t v = (uint32_t)codes[r * count + i];
      for (int t = 0; t < bits; ++t) {
        size_t bit = (size_t)i * bits + t;
        if ((v >> t) & 1u) o[bit >> 3] |= (uint8_t)(1u << (bit & 7));
      }
    }
  }
  return 0;
}

int orc_unpack(const uint8_t* in, int64_t rows, int count, int bits, int32_t* codes) {
  if (bits < 1 || bits > 32) return 1;
  size_t stride = ((size_t)count * bits + 7) / 8;
  for (int64_t r = 0; r < rows; ++r) {
    const uint8_t* p = in + (size_t)r * stride;
    for (int i = 0; i < count; ++i) {
      uint32_t v = 0;
      for (int t = 0; t < bits; ++t) {
        size_t bit = (size_t)i * bits + t;
        v |= (uint32_t)((p[bit >> 3] >> (bit & 7)) & 1u) << t;
      }
      codes[r * count + i] = (int32_t)v;
    }
  }
  return 0;
}

/* Reading R9, record order: slot v of a vector's record (angle and norm codes
 * alike) holds the code of pair phi_d(v).  For d = 64 and 128, with L = d/16:
 *   phi(v) = 4 (v mod L) + ((v / L) mod 4) + 4 L floor(v / 4L),
 * a relabeling of the pair-index bits under which the pairs held by one lane
 * of a kernel that splits a vector over L lanes of 8 pairs (slots l + L m,
 * m = 0..7) are two runs of 4 consecutive pairs.  For d <= 32 the order is
 * the natural one. */
int orc_slot_pair(int d, int v) {
  if (d != 64 && d != 128) return v;
  const int L = d / 16;
  return 4 * (v % L) + (v / L) % 4 + 4 * L * (v / (4 * L));
}

/* Records of `rows` vectors of d/2 codes given in pair order: codes placed in
 * slot order, then packed as orc_pack does. */
int orc_pack_record(const int32_t* codes, int64_t rows, int d, int bits, uint8_t* out) {
  const int P = d / 2;
  int32_t* tmp = (int32_t*)malloc(sizeof(int32_t) * (size_t)P * (size_t)(rows > 0 ? rows : 1));
  if (!tmp) return 2;
  for (int64_t r = 0; r < rows; ++r)
    for (int v = 0; v < P; ++v) tmp[r * P + v] = codes[r * P + orc_slot_pair(d, v)];
  const int rc = orc_pack(tmp, rows, P, bits, out);
  free(tmp);
  return rc;
}

/* The inverse: unpack a record and return its codes in pair order. */
int orc_unpack_record(const uint8_t* in, int64_t rows, int d, int bits, int32_t* codes) {
  const int P = d / 2;
  int32_t* tmp = (int32_t*)malloc(sizeof(int32_t) * (size_t)P * (size_t)(rows > 0 ? rows : 1));
  if (!tmp) return 2;
  int rc = orc_unpack(in, rows, P, bits, tmp);
  if (!rc)
    for (int64_t r = 0; r < rows; ++r)
      for (int v = 0; v < P; ++v) codes[r * P + orc_slot_pair(d, v)] = tmp[r * P + v];
  free(tmp);
  return rc;
}

/* Eq. 1: average angle bits over L layers with per-layer (n_K, n_V). */
double orc_avg_angle_bits(int L, const int* nK, const int* nV) {
  double acc = 0.0;
  for (int l = 0; l < L; ++l) acc += (log2((double)nK[l]) + log2((double)nV[l])) / 4.0;
  return acc / (double)L;
}

/* Eq. 3: total bits per element. */
double orc_total_bits(double b_angle, double b_norm, int d) {
  return b_angle + b_norm / 2.0 + 64.0 / (double)d;
}

/*
 * Attention of nq query vectors over T decoded cache vectors (the consumer of
 * the Sec. 3.1 reconstruction; the paper evaluates its codes through a model's
 * attention, it does not describe a kernel for it):
 *   s_t = scale * (q . k^_t),  p_t = exp(s_t - max_t s_t) / sum_t exp(...),
 *   out = sum_t p_t v^_t
 * with k^_t, v^_t the decoded K and V rows (orc_decode).  Plain fp64.
 *   q     nq x d, khat, vhat  T x d, out  nq x d.  T >= 1.
 */
int orc_attend(const double* q, int nq, const double* khat, const double* vhat, int64_t T, int d,
               double scale, double* out) {
  if (nq < 1 || T < 1 || d < 1) return 1;
  double* s = (double*)malloc(sizeof(double) * (size_t)T);
  if (!s) return 2;
  for (int a = 0; a < nq; ++a) {
    const double* qa = q + (size_t)a * d;
    double mx = -INFINITY;
    for (int64_t t = 0; t < T; ++t) {
      double acc = 0.0;
      for (int j = 0; j < d; ++j) acc += qa[j] * khat[(size_t)t * d + j];
      s[t] = scale * acc;
      if (s[t] > mx) mx = s[t];
    }
    double den = 0.0;
    for (int64_t t = 0; t < T; ++t) {
      s[t] = exp(s[t] - mx);
      den += s[t];
    }
    double* o = out + (size_t)a * d;
    for (int j = 0; j < d; ++j) o[j] = 0.0;
    for (int64_t t = 0; t < T; ++t) {
      const double p = s[t] / den;
      for (int j = 0; j < d; ++j) o[j] += p * vhat[(size_t)t * d + j];
    }
  }
  free(s);
  return 0;
}
