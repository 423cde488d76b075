// TurboAngle encode kernel for sm_103a (Alg. 1 + Sec. 3.3 / Eq. 2 of arXiv 2603.27467).
//
// One kernel per (d, input dtype, n = 2^W, norm bits B, norm mode): a launch
// encodes a batch of jobs that share the codebook shape, so every record size
// is a compile-time constant and the instruction footprint is one body.
//
// Work is split into warp tiles: L = d/16 lanes share a row, each lane owns 8
// angle pairs (16 elements), so a warp encodes RW = 32/L rows at a time.  Every
// warp runs its own pipeline (no block-wide barrier in the main loop):
//   1. a kNS-stage cp.async ring stages its warp tiles global -> shared
//      (coalesced 16-byte chunks, padded rows);
//   2. D is a sign XOR on the raw input bits.  The unnormalized Walsh-Hadamard
//      butterfly runs in two register phases on packed fp32 pairs (FADD2/FFMA2):
//      phase A over the pair-index bits held in registers (lane l holds pairs
//      l + L*m), an intra-warp shared-memory transpose, phase B over the low
//      bits (lane l then holds pairs 8l..8l+7).  The element-pair stage (input
//      bit 0) is never executed: for output pair i the butterfly halves
//      E_i = WHT_i(x_even), O_i = WHT_i(x_odd) give (y_2i, y_2i+1) = (E+O, E-O),
//      so r_i^2 = 2 (E_i^2 + O_i^2) / d and the angle test works on (E_i, O_i);
//   3. Alg. 1's k_i = floor(n theta/2pi + 1/2) mod n is decided by an exact edge
//      test: a candidate edge from an arctangent approximation (the angle of
//      (|E|, |O|) is pi/4 + atan((|O| - |E|) / (|O| + |E|)), with an odd cubic
//      for atan on [-1, 1], max error 0.00496 rad), then the sign of the cross
//      product of (E, O) with the edge direction.  The test is certified by a
//      bound on the fp32 error;
//   4. Eq. 2 norm codes (linear, or on log2 r) against the row's minimum and
//      maximum pair norms, certified the same way against a band around each
//      rounding midpoint; the fp32 extremes are stored as the header
//      (r_min, r_max);
//   5. each lane packs its 8 codes LSB-first; the warp stages its records in
//      shared memory and writes them with one 16-byte store per lane (contiguous
//      slots) or per row (scatter-append slots);
//   6. the codes not certified (about 4e-4 of them) go to a per-warp queue in
//      shared memory, moved to a queue in the call's workspace when it fills;
//      a fix-up kernel after the encode re-decides them (a double-float second
//      look, then exact integer sums of the row) and patches the records.
#include <algorithm>
#include <atomic>

#include "tac_common.cuh"

namespace tac {

// Edge directions (cos psi_e, sin psi_e) for every supported n as double-float
// pairs (c_hi, c_lo, s_hi, s_lo), built in fp64 by the host compiler and read
// warp-uniformly by the exact path.
namespace cx {
struct DfEdgeTable { float4 v[kTabEntries]; };
constexpr DfEdgeTable make_df_edge_table() {
  DfEdgeTable t{};
  for (int idx = 0; idx < kTabEntries; ++idx) {
    const int n = tab_n_of(idx), e = idx - tab_offset_n(n);
    const CS cs = cos_sin_q8(8 * e + 4 + n, n);
    const float ch = (float)cs.c, sh = (float)cs.s;
    t.v[idx] = float4{ch, (float)(cs.c - (double)ch), sh, (float)(cs.s - (double)sh)};
  }
  return t;
}
}  // namespace cx
__constant__ cx::DfEdgeTable g_edge_df = cx::make_df_edge_table();

constexpr int kNS = 4;  // pipeline stages per warp: kNS - 1 warp tiles in flight
constexpr int kQ = 96;  // entries of a warp's re-decision queue
// CTA shape of the encode: 8 warps, two CTAs per SM (16 warps, up to 128
// registers a thread).  10-warp CTAs (up to 96 registers) issued about 3 %
// faster before the re-decision queue, whose bookkeeping no longer fits in 96
// registers without spills in the main loop.
constexpr int kEncWarps = 8;
constexpr int kEncThreads = 32 * kEncWarps;

// Shape of one kernel: n bins (W = ceil(log2 n) bits per angle code), B norm
// bits (4, 8, or 32 for fp32 norms), MODE; HB header bytes per row (8, none
// for fp32 norms).
template <int D, typename TIn, int N, int B, int MODE>
struct Enc {
  using G = Geo<D>;
  using IT = RowTile<D, (int)sizeof(TIn)>;
  static constexpr int P = G::P, L = G::L, RW = G::RW;
  static constexpr int ESZ = (int)sizeof(TIn);
  static constexpr int n = N;
  static constexpr int W = code_bits(N);
  static constexpr int AB = P * W / 8;        // angle record bytes per row
  static constexpr int NB = P * B / 8;        // norm record bytes per row
  static constexpr int HB = (MODE == TAC_NORM_FP32) ? 0 : 8;
  // A warp tile's records: RW*AB = 32 W and RW*NB = 32 B bytes, RW*HB header
  // bytes: every segment is a whole number of 16-byte chunks.
  static constexpr int NA = RW * AB / 16, NN = RW * NB / 16, NH = RW * HB / 16;
  static constexpr int NCH = NA + NN + NH;
  static constexpr int ROUNDS = (NCH + 31) / 32;
  // Input chunk map: 32 consecutive 16-byte chunks cover RPQ rows.
  static constexpr int CPR = IT::CPR, RPQ = 32 / CPR, CHUNKS = IT::CHUNKS;
  // per-warp shared memory region
  static constexpr int W_IN = 0;                            // kNS input stages
  static constexpr int W_TP = W_IN + kNS * IT::BYTES;       // transpose rows
  static constexpr int W_ANG = W_TP + G::TP_W;              // staged records: angle | norm | header
  static constexpr int W_NRM = W_ANG + RW * AB;
  static constexpr int W_HDR = W_NRM + RW * NB;
  static constexpr int W_JOB = W_HDR + RW * HB;             // current job (WarpJob)
  static constexpr int W_RC = W_JOB + 64;                    // the rows' fp32 (smin, smax, ty) for the queue
  static constexpr int W_Q = W_RC + RW * 16;                 // re-decision queue (kQ entries of 32 bytes)
  static constexpr int WARP_B = W_Q + kQ * 32;
  static constexpr int TABR = tab_copies(n, 8192);           // edge table copies
  static constexpr int OFF_TAB = kEncWarps * WARP_B;           // fp32 edge table of this n (TABR copies)
  static constexpr int SMEM = OFF_TAB + n * TABR * 8;
  static_assert((RW * AB) % 16 == 0 && (RW * NB) % 16 == 0 && (RW * HB) % 16 == 0, "record segments");
  static_assert(W_TP % 16 == 0 && W_ANG % 16 == 0 && W_JOB % 16 == 0 && WARP_B % 16 == 0, "alignment");
  static_assert(32 % CPR == 0 && RW % RPQ == 0, "chunk map");
};

// The job a warp is encoding as far as the rare paths need it (exact
// re-decision, tail tiles and scatter), kept in the warp's shared region.
struct WarpJob {
  uint8_t* codes;
  uint8_t* norms;
  uint8_t* hdr;
  const int64_t* slot;
  int64_t capacity;
  uint32_t signs[4];
  int32_t job;         // its index in the launch's job table
};
static_assert(sizeof(WarpJob) <= 64, "WarpJob");

// Store the low NBYTES (<= 8) bytes of (hi:lo) at a shared address aligned to gcd(NBYTES, 8).
template <int NBYTES>
__device__ __forceinline__ void store_bytes(uint8_t* dst, uint32_t lo, uint32_t hi) {
  if constexpr (NBYTES == 8) {
    *reinterpret_cast<uint2*>(dst) = make_uint2(lo, hi);
  } else if constexpr (NBYTES == 4) {
    *reinterpret_cast<uint32_t*>(dst) = lo;
  } else if constexpr (NBYTES % 2 == 0) {
#pragma unroll
    for (int q = 0; q < NBYTES / 2; ++q)
      reinterpret_cast<uint16_t*>(dst)[q] = (uint16_t)((q < 2 ? lo : hi) >> (16 * (q & 1)));
  } else {
#pragma unroll
    for (int q = 0; q < NBYTES; ++q) dst[q] = (uint8_t)((q < 4 ? lo : hi) >> (8 * (q & 3)));
  }
}

// v mod n for v in [-n, 2n).
template <int N>
__device__ __forceinline__ int wrap_bin(int v) {
  if constexpr (is_pow2(N)) return v & (N - 1);
  else return v < 0 ? v + N : (v >= N ? v - N : v);
}

// Candidate edge for the pair (E, O) (butterfly halves, y = (E + O, E - O))
// and n bins, before the reduction mod n: Alg. 1's angle theta = pi/4 -
// angle(E, O) in bins, floored (for n >= 8, M + n/8 - angle rounded down onto
// the integer grid of M = 1.5 * 2^23, where n/8 is an integer and M + n/8
// exact; for n = 2, 4, whose n/8 is not on that grid, a direct conversion
// rounding down, which gives the same value less M).  The
// angle of (|E|, |O|) is pi/4 + atan(t) with t = (|O| - |E|) / (|O| + |E|) in
// [-1, 1], so no octant test is needed; atan(t) ~ t (a + b t^2) is an odd
// cubic fitted minimax on [-1, 1] for this kernel (max error 0.00496 rad).  The
// true bin is the candidate or the next one whenever that error is below half
// a bin, i.e. for every n <= 256 (0.2 bins at n = 256).  A zero pair gives NaN
// here: it is decided by the exact path, and the callers mask or clamp the
// result before it indexes a table.
template <int N>
__device__ __forceinline__ int candidate_bits(float E, float O) {
  constexpr int n = N;
  constexpr float nb = (float)n * 0.15915494309189535f;  // bins per radian
  constexpr float ca = 0.97239412f * nb, cb = -0.19194795f * nb;
  const float aE = fabsf(E), aO = fabsf(O);
  const float t = (aO - aE) * rcp_approx(aO + aE);
  // angle of (|E|, |O|) less n/4, in bins: in [-n/4, 0]
  const float dq = __fmaf_rn(t, __fmaf_rn(t * t, cb, ca), -0.125f * n);
  // angle of (E, |O|): n/4 + dq, or n/2 - (n/4 + dq) = n/4 - dq when E < 0
  const float fb = 0.25f * n + __uint_as_float(__float_as_uint(dq) ^ (__float_as_uint(E) & 0x80000000u));
  const float ab = __uint_as_float(__float_as_uint(fb) ^ (__float_as_uint(O) & 0x80000000u));
  if constexpr (n % 8 != 0) return __float2int_rd(0.125f * n - ab);
  else return __float_as_int(__fadd_rd(12582912.0f + 0.125f * n, -ab));
}

// The candidate edge in [0, n).
template <int N>
__device__ __forceinline__ int candidate_edge(float E, float O) {
  const int bits = candidate_bits<N>(E, O);
  if constexpr (is_pow2(N)) {
    return bits & (N - 1);
  } else {
    // 0x4B400000 = bits of M; the clamp keeps a zero pair's NaN inside [0, n).
    const int e = wrap_bin<N>(bits - 0x4B400000);
    return (int)min((uint32_t)e, (uint32_t)(N - 1));
  }
}

// Alg. 1 bin of the pair (E, O) for n bins by the edge test: the candidate
// edge, then the sign of the cross product with the edge direction (et: this
// lane's copy of the replicated table, R copies).  Returns k; m = O s - E c is
// the cross product with the sign turned (k is the next bin when m < 0); its
// magnitude is the certification margin, and a pair with m == 0 is never
// certified, so which side the fast path gives it does not matter.
template <int N, int R>
__device__ __forceinline__ uint32_t edge_test(float E, float O, const float2* et, float& m) {
  if constexpr (is_pow2(N)) {
    const int bits = candidate_bits<N>(E, O);
    const float2 dir = et[(bits & (N - 1)) * R];
    m = __fmaf_rn(O, dir.y, -__fmul_rn(E, dir.x));
    return (uint32_t)(bits + (int)(__float_as_uint(m) >> 31)) & (uint32_t)(N - 1);
  } else {
    const int e = candidate_edge<N>(E, O);
    const float2 dir = et[e * R];
    m = __fmaf_rn(O, dir.y, -__fmul_rn(E, dir.x));
    return (uint32_t)wrap_bin<N>(e + (int)(__float_as_uint(m) >> 31));
  }
}

// ---------------------------------------------------------------------------
// Exact path.  The butterfly halves E_i = sum_j +-x_2j and O_i = sum_j +-x_2j+1
// of a pair are sums of exactly representable signed input elements; they are
// formed exactly in 64-bit fixed point (integer adds on the ALU: the FP64 pipe
// of this part is too slow for a path that runs on a few rows in a hundred)
// and the decisions are then taken in double-float arithmetic (pairs of fp32,
// about 46 significant bits).
// ---------------------------------------------------------------------------

// One input element (bf16 or fp32 bits), D and its own sign applied, as a
// 64-bit fixed-point number on the scale of the row's largest exponent field
// emax: element = X 2^(emax - K - bias).  K = 47 (bf16) or 31 (fp32) leaves
// room for the sum of d/2 terms; an element more than 2^K below the largest
// loses its bits below the scale (each sum then within d/2 2^-K of the
// largest element).
template <typename TIn>
__device__ __forceinline__ long long fix_elem(uint32_t bits, int emax, uint32_t neg) {
  constexpr bool BF = sizeof(TIn) == 2;
  constexpr int MB = BF ? 7 : 23, K = BF ? 47 : 31;
  const int e = (int)((bits >> MB) & 0xFFu);
  const uint32_t m = (bits & ((1u << MB) - 1u)) | (e != 0 ? (1u << MB) : 0u);
  const int sh = max(e, 1) - emax + K;
  long long x = sh >= 0 ? ((long long)m << sh) : (sh > -(MB + 1) ? (long long)(m >> -sh) : 0ll);
  return neg ? -x : x;
}

// ---- double-float arithmetic (x + y, |y| <= ulp(x)/2) ----
__device__ __forceinline__ float2 df_fast2sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  return make_float2(s, __fadd_rn(b, __fsub_rn(a, s)));
}
__device__ __forceinline__ float2 df_add(float2 a, float2 b) {
  const float s = __fadd_rn(a.x, b.x);
  const float bb = __fsub_rn(s, a.x);
  const float e = __fadd_rn(__fsub_rn(a.x, __fsub_rn(s, bb)), __fsub_rn(b.x, bb));
  return df_fast2sum(s, __fadd_rn(e, __fadd_rn(a.y, b.y)));
}
__device__ __forceinline__ float2 df_neg(float2 a) { return make_float2(-a.x, -a.y); }
__device__ __forceinline__ float2 df_mul(float2 a, float2 b) {
  const float p = __fmul_rn(a.x, b.x);
  float e = __fmaf_rn(a.x, b.x, -p);
  e = __fmaf_rn(a.x, b.y, __fmaf_rn(a.y, b.x, e));
  return df_fast2sum(p, e);
}
__device__ __forceinline__ float2 df_mulf(float2 a, float b) {
  const float p = __fmul_rn(a.x, b);
  return df_fast2sum(p, __fmaf_rn(a.y, b, __fmaf_rn(a.x, b, -p)));
}
__device__ __forceinline__ float2 df_div(float2 a, float2 b) {
  const float r = rcp_approx(b.x);                       // b.x normal and nonzero at every caller
  const float q1 = __fmul_rn(a.x, r);
  const float2 res = df_add(a, df_neg(df_mulf(b, q1)));  // a - q1 b
  return df_fast2sum(q1, __fmul_rn(res.x, r));
}
__device__ __forceinline__ float2 df_sqrt(float2 a) {
  if (!(a.x > 0.f)) return make_float2(0.f, 0.f);
  const float r = sqrt_approx(a.x);
  const float d = __fadd_rn(__fmaf_rn(-r, r, a.x), a.y);
  return df_fast2sum(r, __fmul_rn(d, 0.5f * rcp_approx(r)));
}
__device__ __forceinline__ int df_sign(float2 a) {
  const float v = a.x != 0.f ? a.x : a.y;
  return v > 0.f ? 1 : (v < 0.f ? -1 : 0);
}
// a < b for normalized double-floats (|lo| <= ulp(hi) / 2, as every
// operation here returns them): the leading parts decide unless equal.
__device__ __forceinline__ bool df_less(float2 a, float2 b) { return a.x < b.x || (a.x == b.x && a.y < b.y); }
// 2^k for -126 <= k <= 127, and x 2^k for results in the normal range.
__device__ __forceinline__ float pow2i(int k) { return __uint_as_float((uint32_t)(127 + k) << 23); }
__device__ __forceinline__ float2 df_scale(float2 a, int k) {   // a 2^k, |k| <= 126, normal results
  const float f = pow2i(k);
  return make_float2(a.x * f, a.y * f);
}

// A 64-bit integer as a double-float (its top 48 significant bits; exact below 2^48).
__device__ __forceinline__ float2 ll_to_df(long long v) {
  if (v == 0) return make_float2(0.f, 0.f);
  const bool neg = v < 0;
  const unsigned long long u = neg ? (unsigned long long)(-v) : (unsigned long long)v;
  const int lz = __clzll((long long)u);
  const unsigned long long w = u << lz;                  // leading one at bit 63
  const float hi = (float)(uint32_t)(w >> 40) * pow2i(40 - lz);             // 24 bits: exact
  const float lo = (float)(uint32_t)((w >> 16) & 0xFFFFFFull) * pow2i(16 - lz);
  return neg ? make_float2(-hi, -lo) : make_float2(hi, lo);
}

// Pair energy E^2 + O^2 in double-float from the exact sums.
__device__ __forceinline__ float2 df_energy(longlong2 eo) {
  const float2 e = ll_to_df(eo.x), o = ll_to_df(eo.y);
  return df_add(df_mul(e, e), df_mul(o, o));
}

// Exact angle code (Alg. 1) of a pair from its exact sums: the candidate edge
// from the fp32 polynomial on the leading parts, then the edge test
// m = E cos psi - O sin psi in double-float against the double-float edge
// direction (the code is the next bin when m >= 0).
template <int N>
__device__ __noinline__ int fix_angle_code(longlong2 eo) {
  if (eo.x == 0 && eo.y == 0) return 0;  // pair (0, 0) -> bin 0
  const float2 e = ll_to_df(eo.x), o = ll_to_df(eo.y);
  const int ec = candidate_edge<N>(e.x, o.x);
  const float4 dir = g_edge_df.v[tab_offset_n(N) + ec];
  const float2 m = df_add(df_mul(e, make_float2(dir.x, dir.y)), df_neg(df_mul(o, make_float2(dir.z, dir.w))));
  return wrap_bin<N>(ec + (df_sign(m) >= 0 ? 1 : 0));
}

// log2 of a double-float >= 1, to about 2e-7 absolute: exponent plus log2 of
// the leading part's significand plus the first-order term of the tail.
__device__ __forceinline__ float df_log2_est(float2 a) {
  const int e = (int)((__float_as_uint(a.x) >> 23) & 0xFFu) - 127;
  const float mh = a.x * pow2i(-e), ml = a.y * pow2i(-e);
  return (float)e + log2f(mh) + ml / mh * 1.4426950408889634f;
}

// The exponent of a positive normal fp32 number.
__device__ __forceinline__ int f32_exp(float x) { return (int)((__float_as_uint(x) >> 23) & 0xFFu) - 127; }

// a^n for a double-float a >= 1 and n >= 0, as m 2^e with m in [1, 2) (a
// double-float) and an integer e: every product is brought back to [1, 2),
// so nothing overflows for any n the codes need (n <= 2 * 255 + 1).
__device__ __forceinline__ void df_pow(float2 a, int n, float2& m, int& e) {
  int eb = f32_exp(a.x);
  float2 b = df_scale(a, -eb);
  m = make_float2(1.f, 0.f);
  e = 0;
  while (n) {
    if (n & 1) {
      m = df_mul(m, b);
      e += eb;
      const int k = f32_exp(m.x);
      m = df_scale(m, -k);
      e += k;
    }
    n >>= 1;
    if (n) {
      b = df_mul(b, b);
      eb *= 2;
      const int k = f32_exp(b.x);
      b = df_scale(b, -k);
      eb += k;
    }
  }
}

// rho1^n1 >= rho2^n2 for double-floats rho >= 1 and n >= 0.
static __device__ __noinline__ bool df_pow_ge(float2 r1, int n1, float2 r2, int n2) {
  float2 m1, m2;
  int e1, e2;
  df_pow(r1, n1, m1, e1);
  df_pow(r2, n2, m2, e2);
  if (e1 != e2) return e1 > e2;                          // both significands in [1, 2)
  return !df_less(m1, m2);
}

// Eq. 2 code of a pair from double-float energies s = E^2 + O^2 (unnormalized:
// r^2 = 2 s / d, a common factor that cancels): the pair's (sa) and the row's
// minimum and maximum.  Linear: Lq (r - r_min) / (r_max - r_min); log-space:
// the same on log2 r with norms floored at 2^-24 r_max (log2 r = (log2 s +
// log2(2/d)) / 2: the ratio is taken on the energies); rounded half up and
// clamped; 0 when r_max = r_min (Sec. 3.3, Eq. 2 and its log-space variant).
// A code is c = max{c : the value >= c - 1/2}; an estimate (double-float
// for linear, log2 estimates for log-space) gives c, and only when it lies
// too close to a boundary for its own error is that boundary tested exactly:
// linear by the sign of Lq (r - r_min) - (c - 1/2)(r_max - r_min) in
// double-float; log-space by (s/s_lo)^(2 Lq) >= (s_max/s_lo)^(2c - 1), the
// same inequality raised to integer powers.
template <int B, int MODE>
__device__ __noinline__ int fix_norm_code(float2 sa, float2 smn, float2 smx) {
  constexpr int Lq = (1 << B) - 1;
  int c;
  if constexpr (MODE == TAC_NORM_LINEAR) {
    const float2 a = df_sqrt(sa), m = df_sqrt(smn), M = df_sqrt(smx);
    const float2 A = df_add(a, df_neg(m)), R = df_add(M, df_neg(m));
    if (!(R.x > 0.f)) return 0;                          // r_max = r_min
    auto at_least = [&](int cc) {                        // value >= cc - 1/2
      return df_sign(df_add(df_mulf(A, (float)Lq), df_neg(df_mulf(R, (float)cc - 0.5f)))) >= 0;
    };
    const float2 w = df_add(df_div(df_mulf(A, (float)Lq), R), make_float2(0.5f, 0.f));
    c = (int)floorf(w.x);
    const float fr = __fadd_rn(__fsub_rn(w.x, (float)c), w.y);   // the double-float value is good to 1e-9
    if (fr > 1e-6f && fr < 1.f - 1e-6f) return min(max(c, 0), Lq);
    c = min(max(c, 0), Lq);
    while (c > 0 && !at_least(c)) --c;
    while (c < Lq && at_least(c + 1)) ++c;
  } else {
    const float2 fl = df_scale(smx, -48);                // (2^-24 r_max)^2
    const float2 lo = df_less(smn, fl) ? fl : smn;
    const float2 aa = df_less(sa, fl) ? fl : sa;
    if (!df_less(lo, smx)) return 0;                     // r_max = r_lo
    const float2 r1 = df_div(aa, lo), r2 = df_div(smx, lo);   // >= 1
    auto at_least = [&](int cc) { return df_pow_ge(r1, 2 * Lq, r2, 2 * cc - 1); };
    const float l2 = df_log2_est(r2);
    const float v = __fmaf_rn((float)Lq, df_log2_est(r1) / l2, 0.5f);
    c = (int)floorf(v);
    const float fr = v - (float)c;
    const float tol = (float)Lq * 1e-6f / l2 + 1e-5f;      // the two estimates are good to 2e-7 each
    if (fr > tol && fr < 1.f - tol) return min(max(c, 0), Lq);
    c = min(max(c, 0), Lq);
    while (c > 0 && !at_least(c)) --c;
    while (c < Lq && at_least(c + 1)) ++c;
  }
  return c;
}

// Set bits [bit, bit + w) (w <= 8) of the byte stream at base to code, in
// global memory.  Atomic on the aligned words they touch, so lanes that patch
// different codes of one word do not lose each other's bits.
__device__ __forceinline__ void patch_bits(uint8_t* base, int bit, int w, uint32_t code) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(base) + (uintptr_t)(bit >> 3);
  uint32_t* word = reinterpret_cast<uint32_t*>(a & ~(uintptr_t)3);
  const int sh = (int)(a & 3u) * 8 + (bit & 7);
  const int n0 = min(w, 32 - sh);
  const uint32_t m0 = ((1u << n0) - 1u) << sh;
  atomicAnd(word, ~m0);
  atomicOr(word, (code << sh) & m0);
  if (n0 < w) {
    const uint32_t m1 = (1u << (w - n0)) - 1u;
    atomicAnd(word + 1, ~m1);
    atomicOr(word + 1, (code >> n0) & m1);
  }
}

// ---------------------------------------------------------------------------
// Re-decision queue.  The main loop only notes the codes its bands could not
// settle (a few in ten thousand); each warp keeps them in a queue in its
// shared memory and works through it between tiles when it fills up, and at
// the end.  Doing so outside the tile body keeps the body's registers and
// instructions free of the rare path; the records, written already, are
// patched in place.  An entry (32 bytes): job | slot << 8 | kind << 14, the
// row in the job, then for an angle code the pair's fp32 butterfly halves E, O
// and (in the second half) the row's ty, for a norm code its pair energy s and
// the row's smin, smax and ty of the fast path.  kind: 0 an angle code, 1 a
// norm code, 2 the whole row (rows with more flagged codes than kRowEntries,
// or whose norm band is too wide to be useful).
// ---------------------------------------------------------------------------
template <int D>
struct QGeo {
  static constexpr int RW = Geo<D>::RW;
  static constexpr int kRowEntries = (32 / RW) > 1 ? 32 / RW : 1;   // per row before it goes whole
  static constexpr int kMaxPerTile = RW * kRowEntries;              // <= 32
};

// The part of the norm band left once the fast path's own arithmetic is taken
// out: kKappa times the first-order bound of the transform (see tile_body).
template <int D>
__device__ __forceinline__ constexpr float norm_kappa() { return D >= 64 ? 0.015625f : 0.25f; }

// Second look at a flagged norm code from the fast path's own fp32 values
// (pair energy s, the row's smin, smax and ty) in double-float arithmetic, so
// that only the transform's error is left.  Returns the code when the Eq. 2
// value lies farther than norm_kappa() times that bound from a rounding
// midpoint, else -1.
template <int D, int B, int MODE>
__device__ __noinline__ int norm_second_look(float s, float smin, float smax, float ty) {
  constexpr int Lq = (1 << B) - 1;
  constexpr float kappa = norm_kappa<D>();
  if constexpr (MODE == TAC_NORM_LINEAR) {
    const float2 m = df_sqrt(make_float2(smin, 0.f)), M = df_sqrt(make_float2(smax, 0.f));
    const float2 R = df_add(M, df_neg(m));
    if (!(R.x > 0.f)) return -1;
    // every sqrt(s) within ty; the double-float arithmetic adds far less than 1e-9 Lq
    const float band = kappa * 2.f * (float)Lq * ty / R.x * 1.0001f + 1e-9f * (float)Lq;
    const float2 A = df_add(df_sqrt(make_float2(s, 0.f)), df_neg(m));
    const float2 w = df_add(df_div(df_mulf(A, (float)Lq), R), make_float2(0.5f, 0.f));
    float c = floorf(w.x);
    if (w.x == c && w.y < 0.f) c -= 1.f;
    const float fr = __fadd_rn(__fsub_rn(w.x, c), w.y);
    if (!(fminf(fr, 1.f - fr) > band)) return -1;
    return min(max((int)c, 0), Lq);
  } else {
    const float sfl = smax * 3.5527136788005009e-15f;  // 2^-48 s_max
    const float slo = fmaxf(smin, sfl), sa = fmaxf(s, sfl);
    if (!(smax > slo)) return -1;
    const float l2 = df_log2_est(df_div(make_float2(smax, 0.f), make_float2(slo, 0.f)));
    const float l1 = df_log2_est(df_div(make_float2(sa, 0.f), make_float2(slo, 0.f)));
    // log2 s moves by 2 dsqrt(s) / (sqrt(s) ln 2); each log2 estimate adds 2e-7
    const float band = kappa * 2.f * 1.4426950408889634f * (float)Lq * ty / l2 * 1.01f *
                           (rcp_approx(sqrt_approx(sa)) + rcp_approx(sqrt_approx(slo))) +
                       (float)Lq * (4e-7f / l2 + 8.f * kU);
    const float v = (float)Lq * l1 / l2 + 0.5f;
    const float c = floorf(v);
    const float fr = v - c;
    if (!(fminf(fr, 1.f - fr) > band)) return -1;
    return min(max((int)c, 0), Lq);
  }
}

// Second look at a flagged angle code from the fast path's fp32 butterfly
// halves (E, O) and the row's transform bound ty: the edge test in
// double-float against the double-float edge direction, so that only the
// transform's error is left.  That error moves m = E cos psi - O sin psi by at
// most sqrt(dE^2 + dO^2) <= ty (first order); the code is returned when |m|
// exceeds norm_kappa() of it (the fast band's transform part) plus the
// double-float arithmetic's own (below 2^-43 sqrt(E^2 + O^2)), else -1.  Pairs
// under the fast path's small-norm threshold (same expression, same value)
// always go on to the exact path: their fp32 angle may be off by more than the
// candidate edge allows for.
template <int D, int N>
__device__ __noinline__ int angle_second_look(float E, float O, float ty) {
  const float s = __fmaf_rn(E, E, __fmul_rn(O, O));
  const float rthr = ty * (4.f * (float)N / 3.14159265f);
  if (s < rthr * rthr || !(s > 0.f)) return -1;
  const int ec = candidate_edge<N>(E, O);
  const float4 dir = g_edge_df.v[tab_offset_n(N) + ec];
  const float2 m = df_add(df_mulf(make_float2(dir.x, dir.y), E), df_neg(df_mulf(make_float2(dir.z, dir.w), O)));
  const float band = norm_kappa<D>() * ty * 1.001f + 1.0e-12f * sqrt_approx(s);
  if (!(fabsf(m.x) > band)) return -1;
  return wrap_bin<N>(ec + (m.x > 0.f ? 1 : 0));
}

// The words of one input row a lane takes for the exact path: for pair
// indices jj = lane + 32 q, elements 2 jj and 2 jj + 1 (one 32-bit word of two
// bf16, or two fp32 words).
template <int D, typename TIn>
struct RowWords {
  static constexpr int Q = (Geo<D>::P + 31) / 32;
  static constexpr int NW = sizeof(TIn) == 2 ? Q : 2 * Q;
  uint32_t w[NW];
};

template <int D, typename TIn>
__device__ __forceinline__ void load_row_words(const uint8_t* src, RowWords<D, TIn>& r, int lane) {
  constexpr int P = Geo<D>::P, Q = RowWords<D, TIn>::Q;
#pragma unroll
  for (int q = 0; q < Q; ++q) {
    const int jj = lane + 32 * q;
    if constexpr (sizeof(TIn) == 2) {
      r.w[q] = jj < P ? *reinterpret_cast<const uint32_t*>(src + 4 * jj) : 0u;
    } else {
      const uint2 u = jj < P ? *reinterpret_cast<const uint2*>(src + 8 * jj) : make_uint2(0u, 0u);
      r.w[2 * q] = u.x;
      r.w[2 * q + 1] = u.y;
    }
  }
}

// A lane's elements of one row (pair indices jj = lane + 32 q), D and their
// signs applied, in 64-bit fixed point on the row's largest exponent.
template <int D, typename TIn>
struct FixWords {
  static constexpr int Q = RowWords<D, TIn>::Q;
  long long xe[Q], xo[Q];
};

template <int D, typename TIn>
__device__ __forceinline__ void fix_words(const EncJob& J, const RowWords<D, TIn>& r, FixWords<D, TIn>& f,
                                          int lane) {
  constexpr bool BF = sizeof(TIn) == 2;
  constexpr int P = Geo<D>::P, Q = RowWords<D, TIn>::Q, MB = BF ? 7 : 23, SB = BF ? 15 : 31;
  uint32_t w0[Q], w1[Q];
  int emax = 1;
#pragma unroll
  for (int q = 0; q < Q; ++q) {
    if constexpr (BF) {
      w0[q] = r.w[q] & 0xFFFFu;
      w1[q] = r.w[q] >> 16;
    } else {
      w0[q] = r.w[2 * q];
      w1[q] = r.w[2 * q + 1];
    }
    emax = max(emax, (int)max((w0[q] >> MB) & 0xFFu, (w1[q] >> MB) & 0xFFu));
  }
  emax = (int)__reduce_max_sync(0xffffffffu, (unsigned)emax);
#pragma unroll
  for (int q = 0; q < Q; ++q) {
    const int jj = lane + 32 * q, e0 = 2 * jj, e1 = 2 * jj + 1;
    f.xe[q] = f.xo[q] = 0;
    if (jj < P) {
      const uint32_t s0 = (J.signs[e0 >> 5] >> (e0 & 31)) & 1u, s1 = (J.signs[e1 >> 5] >> (e1 & 31)) & 1u;
      f.xe[q] = fix_elem<TIn>(w0[q], emax, ((w0[q] >> SB) & 1u) ^ s0);
      f.xo[q] = fix_elem<TIn>(w1[q], emax, ((w1[q] >> SB) & 1u) ^ s1);
    }
  }
}

// E and O of the pair in slot v alone, exact (a warp-wide integer sum).
template <int D, typename TIn>
__device__ __forceinline__ longlong2 fix_pair(const FixWords<D, TIn>& f, int v, int lane) {
  constexpr int Q = FixWords<D, TIn>::Q;
  const int ip = slot_pair<D>(v);
  long long e = 0, o = 0;
#pragma unroll
  for (int q = 0; q < Q; ++q) {
    const int jj = lane + 32 * q;
    const bool neg = __popc((unsigned)(ip & jj)) & 1;
    e += neg ? -f.xe[q] : f.xe[q];
    o += neg ? -f.xo[q] : f.xo[q];
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    e += __shfl_xor_sync(0xffffffffu, e, off);
    o += __shfl_xor_sync(0xffffffffu, o, off);
  }
  return make_longlong2(e, o);
}

// Exact butterfly halves of every pair of one row, in 64-bit fixed point in
// the warp's scratch (E at x[0 .. P), O at x[P .. 2P)): the unnormalized
// Sylvester butterfly on the lane's fixed-point elements (integer adds, exact).
template <int D, typename TIn>
__device__ __forceinline__ void exact_row(const FixWords<D, TIn>& f, long long* x, int lane) {
  constexpr int P = Geo<D>::P, Q = FixWords<D, TIn>::Q;
#pragma unroll
  for (int q = 0; q < Q; ++q) {
    const int jj = lane + 32 * q;
    if (jj < P) {
      x[jj] = f.xe[q];
      x[P + jj] = f.xo[q];
    }
  }
  __syncwarp();
#pragma unroll
  for (int lh = 0; (1 << lh) < P; ++lh) {
    const int h = 1 << lh;
#pragma unroll
    for (int q = 0; q < (P + 31) / 32; ++q) {       // P/2 butterflies on each half
      const int bfly = lane + 32 * q;
      if (bfly < P) {
        const int half = bfly / (P / 2), k = bfly % (P / 2);
        const int i0 = half * P + ((k >> lh) << (lh + 1)) + (k & (h - 1));
        const long long a = x[i0], c = x[i0 + h];
        x[i0] = a + c;
        x[i0 + h] = a - c;
      }
    }
    __syncwarp();
  }
}

// Exact minimum and maximum pair energy of the row in scratch (E at x[0, P),
// O at x[P, 2P), 64-bit fixed point) as double-floats, the same on every lane.
// fp32 estimates from the exact sums (each within 4u of its energy, so two
// energies in one order have estimates at most 8 ulp the other way) name the
// candidates: the pairs whose estimate lies within 32 ulp of the smallest
// (largest) estimate.  Only those get the double-float energy.
template <int D>
__device__ __noinline__ void exact_extremes(const long long* x, int lane, float2& smn, float2& smx) {
  constexpr int P = Geo<D>::P, Q = (P + 31) / 32;
  uint32_t eb[Q];
  uint32_t lo = 0xFFFFFFFFu, hi = 0u;
#pragma unroll
  for (int k = 0; k < Q; ++k) {
    const int ip = lane + 32 * k;
    eb[k] = 0u;
    if (ip < P) {
      const float e = __ll2float_rn(x[ip]), o = __ll2float_rn(x[P + ip]);
      eb[k] = __float_as_uint(__fmaf_rn(e, e, __fmul_rn(o, o)));
      lo = min(lo, eb[k]);
      hi = max(hi, eb[k]);
    }
  }
  const uint32_t tmn = __reduce_min_sync(0xffffffffu, lo) + 32u;   // finite estimates: no overflow
  const uint32_t mxb = __reduce_max_sync(0xffffffffu, hi);
  const uint32_t tmx = mxb > 32u ? mxb - 32u : 0u;
  float2 mn = make_float2(3.4028234663852886e38f, 0.f), mx = make_float2(0.f, 0.f);
  bool cmn = false, cmx = false;
#pragma unroll
  for (int k = 0; k < Q; ++k) {
    const int ip = lane + 32 * k;
    if (ip < P && (eb[k] <= tmn || eb[k] >= tmx)) {
      const float2 se = df_energy(make_longlong2(x[ip], x[P + ip]));
      if (eb[k] <= tmn) { cmn = true; if (df_less(se, mn)) mn = se; }
      if (eb[k] >= tmx) { cmx = true; if (df_less(mx, se)) mx = se; }
    }
  }
  const unsigned bmn = __ballot_sync(0xffffffffu, cmn), bmx = __ballot_sync(0xffffffffu, cmx);
  if (__popc(bmn) > 1 || __popc(bmx) > 1) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float2 omn = make_float2(__shfl_xor_sync(0xffffffffu, mn.x, off), __shfl_xor_sync(0xffffffffu, mn.y, off));
      const float2 omx = make_float2(__shfl_xor_sync(0xffffffffu, mx.x, off), __shfl_xor_sync(0xffffffffu, mx.y, off));
      if (df_less(omn, mn)) mn = omn;
      if (df_less(mx, omx)) mx = omx;
    }
    smn = mn;
    smx = mx;
  } else {
    const int a = __ffs(bmn) - 1, b = __ffs(bmx) - 1;
    smn = make_float2(__shfl_sync(0xffffffffu, mn.x, a), __shfl_sync(0xffffffffu, mn.y, a));
    smx = make_float2(__shfl_sync(0xffffffffu, mx.x, b), __shfl_sync(0xffffffffu, mx.y, b));
  }
}

// Works through qn entries of the queue (all lanes of a warp call it), 32 at a
// time, one entry a lane: first the second look at each angle and norm code;
// then, warp-wide and a row at a time, the exact transform of every row that
// still has codes left (a row's entries are consecutive in the queue), from
// which each lane takes its entry's exact sums and the row's exact extreme
// energies; last, each lane decides its own code.  The records in global
// memory are patched.  scratch: 2P longs of the warp's shared memory.
template <int D, typename TIn, int N, int B, int MODE>
__device__ __forceinline__ void flush_queue(const EncJob* jobs, const uint4* q, int qn, long long* scratch, int lane) {
  constexpr int P = Geo<D>::P;
  constexpr int W = code_bits(N);
  constexpr bool FP32N = MODE == TAC_NORM_FP32;
  constexpr int AB = P * W / 8, NB = P * (FP32N ? 32 : B) / 8;
  auto record = [&](const EncJob& J, long long row, uint8_t*& codes, uint8_t*& norms) -> bool {
    const long long sl = J.slot ? J.slot[row] : row;
    if (sl < 0 || sl >= J.capacity) return false;   // skipped slots get no record
    codes = J.codes + sl * AB;
    norms = J.norms + sl * NB;
    return true;
  };
  auto row_src = [&](const EncJob& J, uint32_t row) {
    return reinterpret_cast<const uint8_t*>(J.x) + (long long)row * J.stride * (long long)sizeof(TIn);
  };
  __syncwarp();
  for (int base = 0; base < qn; base += 32) {
    const int e = base + lane;
    uint4 a = make_uint4(0u, 0u, 0u, 0u), b = a;
    uint32_t kind = 3u;
    if (e < qn) {
      a = q[2 * e];
      b = q[2 * e + 1];
      kind = (a.x >> 14) & 3u;
    }
    const uint32_t ej = a.x & 0xFFu;
    const int v = (int)((a.x >> 8) & 63u);
    // ---- second look ----
    int c = -1;
    if (kind == 0u) {
      c = angle_second_look<D, N>(__uint_as_float(a.z), __uint_as_float(a.w), __uint_as_float(b.y));
    } else if (kind == 1u) {
      if constexpr (!FP32N)
        c = norm_second_look<D, B, MODE>(__uint_as_float(a.z), __uint_as_float(a.w), __uint_as_float(b.x),
                                         __uint_as_float(b.y));
    }
    if (c >= 0) {
      uint8_t *codes, *norms;
      if (record(jobs[ej], (long long)a.y, codes, norms)) {
        if (kind == 0u) patch_bits(codes, v * W, W, (uint32_t)c);
        else patch_bits(norms, v * B, B, (uint32_t)c);
      }
    }
    const bool need = kind != 3u && c < 0;
    const unsigned nm = __ballot_sync(0xffffffffu, need);
    if (nm == 0u) continue;
    // ---- rows left: runs of needed entries of one (job, row) ----
    const unsigned below = nm & ((1u << lane) - 1u);
    const int pl = below ? 31 - __clz(below) : lane;
    const uint32_t pj = __shfl_sync(0xffffffffu, ej, pl), pr = __shfl_sync(0xffffffffu, a.y, pl);
    const bool start = need && (below == 0u || pj != ej || pr != a.y);
    unsigned sm = __ballot_sync(0xffffffffu, start);
    const unsigned upto = sm & (lane == 31 ? 0xFFFFFFFFu : ((2u << lane) - 1u));
    const int mys = need ? 31 - __clz(upto) : -1;     // the lane that starts this lane's row
    longlong2 eo = make_longlong2(0, 0);
    float2 smn = make_float2(0.f, 0.f), smx = make_float2(0.f, 0.f);
    while (sm != 0u) {
      const int rs = __ffs(sm) - 1;
      sm &= sm - 1u;
      const uint32_t rj = __shfl_sync(0xffffffffu, ej, rs), rr = __shfl_sync(0xffffffffu, a.y, rs);
      const EncJob& R = jobs[rj];
      RowWords<D, TIn> rw;
      load_row_words<D, TIn>(row_src(R, rr), rw, lane);
      FixWords<D, TIn> fw;
      fix_words<D, TIn>(R, rw, fw, lane);
      exact_row<D, TIn>(fw, scratch, lane);
      const bool mine = mys == rs;
      float2 rmn = make_float2(0.f, 0.f), rmx = make_float2(0.f, 0.f);
      if constexpr (!FP32N) {
        if (__ballot_sync(0xffffffffu, mine && kind != 0u) != 0u) exact_extremes<D>(scratch, lane, rmn, rmx);
      }
      if (mine) {
        smn = rmn;
        smx = rmx;
        if (kind != 2u) {
          const int ip = slot_pair<D>(v);
          eo = make_longlong2(scratch[ip], scratch[P + ip]);
        }
      }
      if (__ballot_sync(0xffffffffu, mine && kind == 2u) != 0u) {   // the whole row, a pair a lane
        uint8_t *codes, *norms;
        if (record(R, (long long)rr, codes, norms)) {
          for (int ip = lane; ip < P; ip += 32) {
            const longlong2 pe = make_longlong2(scratch[ip], scratch[P + ip]);
            const int vs = pair_slot<D>(ip);
            patch_bits(codes, vs * W, W, (uint32_t)fix_angle_code<N>(pe));
            if constexpr (!FP32N)
              patch_bits(norms, vs * B, B, (uint32_t)fix_norm_code<B, MODE>(df_energy(pe), rmn, rmx));
          }
        }
      }
      __syncwarp();
    }
    // ---- exact decisions, one entry a lane ----
    if (need && kind != 2u) {
      uint8_t *codes, *norms;
      if (record(jobs[ej], (long long)a.y, codes, norms)) {
        if (kind == 0u) {
          patch_bits(codes, v * W, W, (uint32_t)fix_angle_code<N>(eo));
        } else {
          if constexpr (!FP32N) patch_bits(norms, v * B, B, (uint32_t)fix_norm_code<B, MODE>(df_energy(eo), smn, smx));
        }
      }
    }
  }
  __syncwarp();
}

// Moves a warp's qn queued entries to the launch's queue in global memory
// (one atomic add reserves their places).  Entries beyond its capacity set
// their row's bit in ovf instead: the fix-up kernel then re-decides that row
// whole.
template <int D>
__device__ __forceinline__ void spill_queue(const EncParams& p, const uint4* q, int qn, int lane) {
  __syncwarp();
  unsigned long long base = 0;
  if (lane == 0) base = atomicAdd(p.gq_n, (unsigned long long)qn);
  base = __shfl_sync(0xffffffffu, base, 0);
  const unsigned long long cap = (unsigned long long)p.gq_cap;
  const int fit = base >= cap ? 0 : (int)min((unsigned long long)qn, cap - base);
  for (int i = lane; i < 2 * fit; i += 32) p.gq[2 * base + i] = q[i];
  for (int e = fit + lane; e < qn; e += 32) {
    const uint4 a = q[2 * e];
    const long long bit = (long long)p.job[a.x & 0xFFu].tile0 * Geo<D>::RW + a.y;
    atomicOr(p.ovf + (bit >> 5), 1u << (bit & 31));
  }
  __syncwarp();
}

// Encode this lane's 8 pairs of warp-tile row r (lane l of the row) and stage
// the records; N bins, B = norm bits, MODE = TAC_NORM_LINEAR / TAC_NORM_LOG /
// TAC_NORM_FP32 (B = 32: the pair norms themselves, no header).
template <int D, typename TIn, int N, int B, int MODE>
__device__ __forceinline__ void tile_body(const uint8_t* in, uint8_t* wsm, const float2* et, int nrows,
                                          int lane, const uint2 (&msk)[8], uint4* q, int& qn, int t,
                                          const EncParams& p) {
  // bf16: msk[m].x holds the sign bits of the pair's two elements (bits 15
  // and 31), msk[m].y the low element's bit moved to bit 31.  The low element
  // widens as w * 2^16 + msk.y (adding bit 31 is an XOR of it: one integer
  // multiply-add), the high one as (w ^ msk.x) & 0xFFFF0000 (one logic op).
  using C = Enc<D, TIn, N, B, MODE>;
  using G = Geo<D>;
  using IT = typename C::IT;
  constexpr int P = C::P, L = C::L;
  constexpr int n = N, W = C::W;
  constexpr int AB = C::AB, NB = C::NB;
  constexpr bool FP32N = MODE == TAC_NORM_FP32;
  constexpr int Lq = FP32N ? 0 : (1 << B) - 1;
  const int r = lane / L, l = lane % L;
  const bool live = r < nrows;
  static_assert(P == 8 * L, "geometry");

  // ---- load 8 pairs (i = l + L*m), apply D, widen ----
  float2 v[8];
  if constexpr (run_layout<D>()) {
    // slots l + L m: pairs 4l + (m & 3) + 4L (m >> 2), two 16-byte (bf16) or
    // 32-byte (fp32) runs of 4 pairs
    const uint8_t* row = in + r * IT::STRIDE + 8 * C::ESZ * l;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const uint8_t* run = row + h * 8 * C::ESZ * L;
      if constexpr (C::ESZ == 2) {
        const uint4 q = *reinterpret_cast<const uint4*>(run);
        const uint32_t u[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint2 mk = msk[4 * h + j];
          v[4 * h + j] = make_float2(__uint_as_float(u[j] * 65536u + mk.y),
                                     __uint_as_float((u[j] ^ mk.x) & 0xFFFF0000u));
        }
      } else {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          const uint4 q = *reinterpret_cast<const uint4*>(run + 16 * k);
          v[4 * h + 2 * k] = make_float2(__uint_as_float(q.x ^ msk[4 * h + 2 * k].x),
                                         __uint_as_float(q.y ^ msk[4 * h + 2 * k].y));
          v[4 * h + 2 * k + 1] = make_float2(__uint_as_float(q.z ^ msk[4 * h + 2 * k + 1].x),
                                             __uint_as_float(q.w ^ msk[4 * h + 2 * k + 1].y));
        }
      }
    }
  } else {
    const uint8_t* row = in + r * IT::STRIDE + 2 * C::ESZ * l;
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      if constexpr (C::ESZ == 2) {
        const uint32_t u = *reinterpret_cast<const uint32_t*>(row + 4 * L * m);
        v[m] = make_float2(__uint_as_float(u * 65536u + msk[m].y), __uint_as_float((u ^ msk[m].x) & 0xFFFF0000u));
      } else {
        const uint2 u = *reinterpret_cast<const uint2*>(row + 8 * L * m);
        v[m] = make_float2(__uint_as_float(u.x ^ msk[m].x), __uint_as_float(u.y ^ msk[m].y));
      }
    }
  }
  // ---- phase A: butterfly over pair-index bits log2(L)..log2(L)+2 ----
  butterfly8<8>(v);
  if constexpr (L > 1) {
    // ---- transpose within the warp: lane l now owns pairs 8l..8l+7 ----
    uint8_t* tpr = wsm + C::W_TP + r * G::ST;
#pragma unroll
    for (int m = 0; m < 8; ++m) *reinterpret_cast<float2*>(tpr + m * G::SM + 8 * (l ^ G::swa(m))) = v[m];
    __syncwarp();
    const uint8_t* tpl = tpr + (8 / L) * l * G::SM;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 t = *reinterpret_cast<const float4*>(tpl + G::tp_pair((2 * q) ^ G::swb(l)));
      v[2 * q] = make_float2(t.x, t.y);
      v[2 * q + 1] = make_float2(t.z, t.w);
    }
    // ---- phase B: butterfly over pair-index bits 0..log2(L)-1 ----
    butterfly8<L>(v);
  }

  // ---- pass 1: pair energies s_j = E^2 + O^2 (r^2 = 2 s / d), row min/max ----
  float s[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) s[j] = __fmaf_rn(v[j].x, v[j].x, __fmul_rn(v[j].y, v[j].y));
  const float lmin_s = min3(min3(s[0], s[1], s[2]), min3(s[3], s[4], s[5]), fminf(s[6], s[7]));
  float smin = lmin_s;
  float smax = max3(max3(s[0], s[1], s[2]), max3(s[3], s[4], s[5]), fmaxf(s[6], s[7]));
  float ssum = ((s[0] + s[1]) + (s[2] + s[3])) + ((s[4] + s[5]) + (s[6] + s[7]));

  // ---- angle codes (Alg. 1): they need no row constant, so they are decided
  // before the row reductions (whose shuffle latency they cover) ----
  uint32_t alo = 0, ahi = 0;
  float am[8];                                  // |m|: each pair's certification margin
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    float m;
    const uint32_t k = edge_test<N, C::TABR>(v[j].x, v[j].y, et, m);
    am[j] = fabsf(m);
    // fields are disjoint and k < n: the adds are ORs (one IMAD each)
    const int sa = j * W;
    if (sa + W <= 32) alo += k << sa;
    else if (sa >= 32) ahi += k << (sa - 32);
    else { alo += k << sa; ahi += k >> (32 - sa); }
  }

  const float mmin = min3(min3(am[0], am[1], am[2]), min3(am[3], am[4], am[5]), fminf(am[6], am[7]));

  // ---- row min / max / sum over the row's L lanes ----
#pragma unroll
  for (int off = 1; off < L; off <<= 1) {
    smin = fminf(smin, __shfl_xor_sync(0xffffffffu, smin, off));
    smax = fmaxf(smax, __shfl_xor_sync(0xffffffffu, smax, off));
    ssum += __shfl_xor_sync(0xffffffffu, ssum, off);
  }
  const bool zero_row = smax == 0.f;               // (a NaN row goes on, to the non-finite check)

  // ---- row constants: stored header (Sec. 3.3), Eq. 2 as code = floor(f(s) qs + qo) ----
  constexpr float k2 = 2.0f / (float)D;
  constexpr float rk2 = D == 16 ? 0.35355339059327379f : D == 32 ? 0.25f : D == 64 ? 0.17677669529663687f : 0.125f;
  // sqrt(2/d) above.  Exact power-of-two scaling: sigma = 4^-k with
  // smax * sigma in [1, 4) (at least 2^-25 for the smallest subnormal smax), so
  // the square roots and logarithms of the row and of its pairs run on normal
  // arguments in their flush-to-zero hardware forms and are scaled back
  // exactly: sqrt(s) = 2^k sqrt(s sigma), log2 s = log2(s sigma) + 2k.
  const int ek = ((int)((__float_as_uint(smax) >> 23) & 0xFFu) - 127) >> 1;
  const int kk = ek < -62 ? -62 : (ek > 63 ? 63 : ek);
  const float sigma = __uint_as_float((uint32_t)(127 - 2 * kk) << 23);
  const float sr = __uint_as_float((uint32_t)(127 + kk) << 23);   // 2^k
  const float smax_s = smax * sigma;
  // sqrt(smax sigma); for d = 32, 128 the factor 2/d of r^2 is an even power of
  // two, so sqrt(smax sigma 2/d) is taken as this times sqrt(2/d), an exact
  // product (one hardware square root, about 1 ulp, either way).
  constexpr bool kEvenK2 = D == 32 || D == 128;
  const float rms = sqrt_ftz(smax_s);
  float hmin = 0.f, hmax = 0.f, qs = 0.f, qo = 0.f, sfloor = 0.f, sc = 0.f;
  if constexpr (FP32N) {
    // no header: the norms are stored as they are (Sec. 3.1)
  } else if constexpr (MODE == TAC_NORM_LINEAR) {
    hmin = sqrt_approx(smin * k2);              // smin * sigma may still be subnormal
    hmax = (kEvenK2 ? rms * rk2 : sqrt_ftz(smax_s * k2)) * sr;
    sc = (float)Lq * rcp_approx(hmax - hmin);
    qs = sc * rk2;                              // f(s) = sqrt(s)
    qo = __fmaf_rn(-hmin, sc, 0.5f);
    if (!(hmax > hmin) || !(sc <= 3.0e38f)) { qs = 0.f; qo = 0.5f; }
  } else {  // log-space, norms floored at 2^-24 r_max
    sfloor = smax * 3.5527136788005009e-15f;    // 2^-48 on the energy
    const float hmin_s = sqrt_ftz(fmaxf(smin, sfloor) * sigma * k2);   // >= 2^-24 hmax_s: normal
    const float hmax_s = kEvenK2 ? rms * rk2 : sqrt_ftz(smax_s * k2);
    hmin = hmin_s * sr;
    hmax = hmax_s * sr;
    const float lmin_s = lg2_ftz(hmin_s);
    sc = (float)Lq * rcp_approx(lg2_ftz(hmax_s) - lmin_s);
    qs = 0.5f * sc;                             // f(s) = log2 s; log2 r = (log2 s + log2 k2)/2
    qo = __fmaf_rn(0.5f * (float)(G::LOGD == 4 ? -3 : G::LOGD == 5 ? -4 : G::LOGD == 6 ? -5 : -6) -
                       (lmin_s + (float)kk),
                   sc, 0.5f);
    if (!(hmax > hmin) || !(sc <= 3.0e38f)) { qs = 0.f; qo = 0.5f; }
  }
  // Certification bound on the cross product m = E c - O s.  The butterfly's
  // log2 d - 1 rounded stages give |dE| <= (log2 d - 1) u ||x_even||_1 and
  // |dO| <= (log2 d - 1) u ||x_odd||_1 (first order), so with c^2 + s^2 = 1
  //   |dm| <= (log2 d - 1) u sqrt(||x_even||_1^2 + ||x_odd||_1^2)
  //        <= (log2 d - 1) u sqrt(d/2) ||x||_2 = (log2 d - 1) u sqrt(S),
  // S = sum_i (E_i^2 + O_i^2) = d ||x||_2^2 / 2 (the factor 1.01 covers the
  // rounding of the computed S and the second-order terms).  The edge direction
  // (each entry within 1 ulp, i.e. 2u relative) and the product E c (u) add
  // at most 2u (|E||c| + |O||s|) + u |E c| <= 3u sqrt(E^2 + O^2) <= 3u sqrt(smax);
  // the fma's own rounding cannot change the sign of a nonzero result.
  // The same ty bounds the error of every sqrt(E^2 + O^2) (the unnormalized
  // pair norm), so ty sqrt(2/d) bounds the error of each r_i.
  // The angle band takes norm_kappa() of the transform's part (see the norm
  // band below) and all of the arithmetic's part.
  const float rmx = rms * sr;
  const float ty = (float)(G::LOGD - 1) * kU * 1.01f * (sqrt_ftz(ssum * sigma) * sr);
  const float tau = norm_kappa<D>() * ty + 3.03f * kU * rmx;
  // The per-pair norm functions below take s itself (pairs below the log floor
  // are clamped to it first), against the true-scale qs, qo: for inputs in the
  // supported range every nonzero s is a normal fp32 number, so the
  // flush-to-zero hardware forms see it unchanged.
  // Pairs whose norm is so small that the fp32 angle may be off by a quarter bin
  // are re-decided too: sqrt(s) < 4 n ty / pi.
  const float rthr = ty * (4.f * (float)n / 3.14159265f);
  const float sthr = rthr * rthr;
  if (l == 0) reinterpret_cast<float4*>(wsm + C::W_RC)[r] = make_float4(smin, smax, ty, 0.f);

  // Norm-code band (Eq. 2).  The code is floor(t), t = f(s) qs + qo the Eq. 2
  // value plus 1/2; it is re-decided exactly when t lies within th of an
  // integer (a rounding midpoint of Eq. 2).  th adds two parts:
  //  - the butterfly: kKappa times the first-order bound of the fp32 transform
  //    (ty on every pair norm; linear: 2 Lq tau_r / (r_max - r_min), log: the
  //    same on log2 r with 1/r_i <= 1/r_lo, tau_r = ty sqrt(2/d)).  That bound
  //    assumes every rounding of every stage at its maximum and with one sign;
  //    the errors measured on the synthetic caches of every workload stay
  //    below 0.075 of it for a pair norm at d = 64, 128 (0.17 at d <= 32), and
  //    their distribution is what kKappa is set from: in a simulation of the
  //    fp32 transform over 1.3e8 pairs of every workload no norm code (and
  //    over 1.8e8 codes no angle code) decided from the fp32 values outside
  //    the band at kKappa = 1/128 differed from the exact one.  kKappa = 1/64
  //    (d >= 64) or 1/4 (d <= 32) is used.  It is no proof for every input: a
  //    code can still differ where the transform's error exceeds kKappa of its
  //    bound and the exact value lies closer to the midpoint than that error,
  //    i.e. within about 1e-4 code units (or 1e-7 rad) of it, where the parity
  //    rule counts such codes;
  //  - the kernel's own arithmetic, bounded in full: each computed norm (the
  //    pair's, r_min's, r_max's) within kEr of its value for the computed
  //    energy (hardware square root, rounding of the energy), qs within kEq,
  //    log2 within kEl absolute plus a rounding of the result, and the roundings
  //    of qo and of the final fma at magnitudes up to 2^(B+1).
  // A row whose band reaches 1/4 (rows of nearly equal pair norms, non-finite
  // rows) has every norm code re-decided.
  constexpr float kKappa = norm_kappa<D>();
  // kEr: hardware sqrt <= 2u relative (1 ulp) plus the energy's rounding
  // (2u on s, u on its root); kEq: rcp <= 2u plus two roundings; kEl: lg2
  // <= 2^-22 absolute on [1/2, 2), and within 4u |result| elsewhere (a GPU
  // test checks each of these limits over whole binades).
  constexpr float kEr = 3.f * kU, kEq = 4.f * kU, kEl = 2.384185791015625e-07f;  // 2^-22
  constexpr float kMag = FP32N ? 0.f : (float)(1 << (B & 15));  // 2^B
  constexpr int kFb = 23 - (FP32N ? 8 : B);                     // fraction bits of t + 2^B
  constexpr uint32_t kFracMask = (1u << kFb) - 1u;
  float th = 0.f;
  if constexpr (!FP32N) {
    if constexpr (MODE == TAC_NORM_LINEAR) {
      th = kKappa * 2.f * qs * ty + 2.f * kEr * (hmax + hmin) * sc + (float)Lq * kEq +
           kU * (hmin * sc + 4.f * kMag + 2.f);
    } else {
      const float elp = kEl + 4.f * kU * (fabsf(2.f * (float)kk) + 52.f);   // log2 of one pair's energy
      th = kKappa * 2.f * sc * (ty * rk2) * rcp_approx(hmin) * 1.4426950408889634f + 1.5f * sc * elp +
           (float)Lq * kEq + kU * (fabsf(qo) + 4.f * kMag + 2.f);
    }
  }
  const bool nall = !(th < 0.25f);              // also NaN
  const float thu = nall ? 0.f : th;
  // t + 2^B + th (in [2^B, 2^(B+1))): the integer part of t + th sits in the
  // mantissa bits [23 - B, 23) and its fraction in the kFb bits below
  const float qo2 = qo + (kMag + thu);
  const uint32_t thb2 = nall ? 0xFFFFFFFFu : 2u * ((uint32_t)(thu * (float)(1u << kFb)) + 1u);

  // ---- pass 2: norm codes (Eq. 2), packing ----
  uint32_t nlo = 0, nhi = 0;
  uint32_t nfr = 0xFFFFFFFFu;                   // smallest fraction field of t + th over the lane's pairs
  float rn[FP32N ? 8 : 1];                      // fp32 norms r_j = sqrt(2 s_j / d)
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    if constexpr (FP32N) {
      rn[j] = sqrt_approx(s[j] * k2);
    } else {
      float f;
      if constexpr (MODE == TAC_NORM_LINEAR) f = sqrt_ftz(s[j]);
      else f = lg2_ftz(fmaxf(s[j], sfloor));
      const uint32_t tb = __float_as_uint(__fmaf_rn(f, qs, qo2));
      nfr = min(nfr, tb & kFracMask);
      // code floor(t + th) = bits [kFb, kFb + B) of tb, moved to its field at
      // bit j B (a pair within th of a midpoint is re-decided below)
      const int sn = j * B;
      const int sh = kFb - (sn & 31);
      const uint32_t part = (sh >= 0 ? (tb >> sh) : (tb << -sh)) & ((uint32_t)Lq << (sn & 31));
      if (sn < 32) nlo |= part; else nhi |= part;
    }
  }
  const bool nflag = !FP32N && (nall || nfr < thb2);
  // fl: bits 0-7 name the angle codes to re-decide, bits 8-15 the norm codes
  uint32_t fl = 0;
  // a row whose energy sum is not finite may hold a NaN or an inf: its lanes
  // look at their 16 staged elements
  const bool odd = !(ssum <= 3.4028234663852886e38f);
  bool nf = false;
  if (zero_row) { alo = ahi = nlo = nhi = 0; hmin = hmax = 0.f; }
  else if (mmin < tau || lmin_s < sthr || nflag || odd) {  // rare: name the uncertified pairs
    if (odd) {
      const uint4* e16 = reinterpret_cast<const uint4*>(in + r * IT::STRIDE + l * 16 * C::ESZ);
#pragma unroll
      for (int c = 0; c < C::ESZ; ++c) {
        const uint4 w = e16[c];
        const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          if constexpr (C::ESZ == 2)
            nf |= (ww[k] & 0x7F80u) == 0x7F80u || (ww[k] & 0x7F800000u) == 0x7F800000u;
          else
            nf |= (ww[k] & 0x7F800000u) == 0x7F800000u;
        }
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (am[j] < tau || s[j] < sthr) fl |= 1u << j;
    if constexpr (!FP32N) {
      if (nflag) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          float f;
          if constexpr (MODE == TAC_NORM_LINEAR) f = sqrt_ftz(s[j]);
          else f = lg2_ftz(fmaxf(s[j], sfloor));
          if (nall || (__float_as_uint(__fmaf_rn(f, qs, qo2)) & kFracMask) < thb2) fl |= 0x100u << j;
        }
      }
    }
  }
  if (!live) { fl = 0; nf = false; }

  // ---- rows holding a NaN or an inf: all codes 0, header (NaN, NaN), the
  // job's status word set; then queue the codes to re-decide (kQ - qn >=
  // kMaxPerTile on entry) ----
  if (__ballot_sync(0xffffffffu, fl != 0u || nf) != 0u) {
    using QG = QGeo<D>;
    const unsigned nfb = __ballot_sync(0xffffffffu, nf);
    if (nfb != 0u) {
      constexpr uint32_t kRL = (L >= 32) ? 0xFFFFFFFFu : ((1u << L) - 1u);
      if ((nfb >> (r * L)) & kRL) {
        const float qnan = __int_as_float(0x7FC00000);
        fl = 0;
        alo = ahi = nlo = nhi = 0;
        hmin = hmax = qnan;
        if constexpr (FP32N) {
#pragma unroll
          for (int j = 0; j < 8; ++j) rn[j] = qnan;
        }
        if (l == 0) {
          uint32_t* st = p.job[reinterpret_cast<const WarpJob*>(wsm + C::W_JOB)->job].status;
          if (st) atomicOr(st, (uint32_t)TAC_E_NONFINITE);
        }
      }
    }
    const int cnt = __popc(fl & 0xFFFFu);
    int rowcnt = cnt;
#pragma unroll
    for (int off = 1; off < L; off <<= 1) rowcnt += __shfl_xor_sync(0xffffffffu, rowcnt, off);
    const bool whole = rowcnt > QG::kRowEntries || (nall && rowcnt > 0);
    const int mine = whole ? (l == 0 ? 1 : 0) : cnt;
    int inc = mine;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, inc, off);
      if (lane >= off) inc += o;
    }
    if (mine) {
      uint4* e = q + 2 * (qn + inc - mine);
      const WarpJob* wj = reinterpret_cast<const WarpJob*>(wsm + C::W_JOB);
      const int cj = wj->job;
      const uint32_t row = (uint32_t)((long long)(t - p.job[cj].tile0) * C::RW + r);
      const uint32_t hd = (uint32_t)cj;
      const float4 rc = reinterpret_cast<const float4*>(wsm + C::W_RC)[r];
      if (whole) {
        e[0] = make_uint4(hd | (2u << 14), row, 0u, 0u);
        e[1] = make_uint4(0u, 0u, 0u, 0u);
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if ((fl >> j) & 1u) {
            e[0] = make_uint4(hd | ((uint32_t)(8 * l + j) << 8), row, __float_as_uint(v[j].x),
                              __float_as_uint(v[j].y));
            e[1] = make_uint4(0u, __float_as_uint(ty), 0u, 0u);
            e += 2;
          }
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if ((fl >> (8 + j)) & 1u) {
            e[0] = make_uint4(hd | ((uint32_t)(8 * l + j) << 8) | (1u << 14), row, __float_as_uint(s[j]),
                              __float_as_uint(rc.x));
            e[1] = make_uint4(__float_as_uint(rc.y), __float_as_uint(rc.z), 0u, 0u);
            e += 2;
          }
        }
      }
    }
    qn += __shfl_sync(0xffffffffu, inc, 31);
  }

  // ---- stage the records ----
  if (live) {
    store_bytes<W>(wsm + C::W_ANG + r * AB + l * W, alo, ahi);
    if constexpr (FP32N) {
      float4* dst = reinterpret_cast<float4*>(wsm + C::W_NRM + r * NB + l * 32);
      dst[0] = make_float4(rn[0], rn[1], rn[2], rn[3]);
      dst[1] = make_float4(rn[4], rn[5], rn[6], rn[7]);
    } else {
      store_bytes<B>(wsm + C::W_NRM + r * NB + l * B, nlo, nhi);
      if (l == 0) reinterpret_cast<float2*>(wsm + C::W_HDR)[r] = make_float2(hmin, hmax);
    }
  }
  __syncwarp();

}

// Records of a tail tile (nrows < RW) or of scattered slots, from the staged
// records to the planes.
template <int AB, int NB, int HB>
__device__ __noinline__ void copy_out_slow(const WarpJob* wj, const uint8_t* sang, const uint8_t* snrm,
                                           const uint8_t* shdr, int64_t row0, int nrows, int lane) {
  if (wj->slot == nullptr) {
    uint8_t* ga = wj->codes + row0 * AB;
    uint8_t* gn = wj->norms + row0 * NB;
    uint8_t* gh = wj->hdr + row0 * 8;
    for (int q = lane; q < nrows * AB; q += 32) ga[q] = sang[q];
    for (int q = lane; q < nrows * NB; q += 32) gn[q] = snrm[q];
    if constexpr (HB > 0)
      for (int q = lane; q < nrows * HB; q += 32) gh[q] = shdr[q];
  } else if (lane < nrows) {
    const int64_t s = wj->slot[row0 + lane];
    if (s < 0 || s >= wj->capacity) return;  // out-of-range slots are skipped
    uint8_t* ga = wj->codes + s * AB;
    uint8_t* gn = wj->norms + s * NB;
    const uint8_t* a = sang + lane * AB;
    const uint8_t* nn = snrm + lane * NB;
    if constexpr ((AB & 15) == 0) {
      for (int q = 0; q < AB / 16; ++q) reinterpret_cast<uint4*>(ga)[q] = reinterpret_cast<const uint4*>(a)[q];
    } else if constexpr ((AB & 7) == 0) {
      for (int q = 0; q < AB / 8; ++q) reinterpret_cast<uint2*>(ga)[q] = reinterpret_cast<const uint2*>(a)[q];
    } else if constexpr ((AB & 3) == 0) {
      for (int q = 0; q < AB / 4; ++q) reinterpret_cast<uint32_t*>(ga)[q] = reinterpret_cast<const uint32_t*>(a)[q];
    } else {
      for (int q = 0; q < AB; ++q) ga[q] = a[q];
    }
    if constexpr ((NB & 7) == 0) {
      for (int q = 0; q < NB / 8; ++q) reinterpret_cast<uint2*>(gn)[q] = reinterpret_cast<const uint2*>(nn)[q];
    } else {
      for (int q = 0; q < NB / 4; ++q) reinterpret_cast<uint32_t*>(gn)[q] = reinterpret_cast<const uint32_t*>(nn)[q];
    }
    if constexpr (HB > 0) reinterpret_cast<float2*>(wj->hdr)[s] = reinterpret_cast<const float2*>(shdr)[lane];
  }
}

template <int D, typename TIn, int N, int B, int MODE>
// Two CTAs of kEncWarps warps per SM (see kEncWarps).
__global__ void __launch_bounds__(kEncThreads, kMinBlocks) encode_kernel(const __grid_constant__ EncParams p) {
  using C = Enc<D, TIn, N, B, MODE>;
  using IT = typename C::IT;
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;

  // fp32 edge table of this n (shared by the CTA).
  float2* etab = reinterpret_cast<float2*>(smem + C::OFF_TAB);
  for (int e = tid; e < C::n; e += kEncThreads) {
    const float2 cs = cos_sin_q8(edge_q8(e, C::n), C::n);
#pragma unroll
    for (int c = 0; c < C::TABR; ++c) etab[e * C::TABR + c] = cs;
  }
  // the job table, for the fix-up kernel
  if (blockIdx.x == 0) {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(p.job);
    uint32_t* dst = reinterpret_cast<uint32_t*>(p.gjobs);
    const int words = p.njobs * (int)(sizeof(EncJob) / 4);
    for (int i = tid; i < words; i += kEncThreads) dst[i] = src[i];
  }
  __syncthreads();

  // Each warp owns a contiguous range of warp tiles (balanced to +-1 tile), so
  // it meets a new job at most a few times per launch and walks its planes
  // with pointer increments.
  const int Gw = gridDim.x * kEncWarps, gw = blockIdx.x * kEncWarps + warp;
  const int per = p.ntiles / Gw, extra = p.ntiles % Gw;
  int t = gw * per + min(gw, extra);
  const int t_end = t + per + (gw < extra ? 1 : 0);
  if (t >= t_end) return;
  uint8_t* wsm = smem + warp * C::WARP_B;

  // ---- prefetch cursor: the next warp tile to load ----
  // Lane chunk q of a tile is row q*RPQ + lane/CPR, bytes (lane % CPR)*16.
  const int lane_cr = lane / C::CPR;
  uint8_t* const in_dst = wsm + C::W_IN + lane_cr * IT::STRIDE + (lane % C::CPR) * 16;
  int it = t;                    // next tile to issue
  int pj = find_job(p, t);       // its job
  int p_end = 0;                 // first tile after that job
  int64_t i_left = 0;            // rows of the job from the tile's row 0
  int64_t i_step = 0;            // bytes between consecutive tiles (RW rows)
  int64_t i_qstep = 0;           // bytes between a lane's consecutive chunks (RPQ rows)
  const uint8_t* i_src = nullptr;  // this lane's first chunk of the tile
  auto set_issue_job = [&]() {
    const EncJob& J = p.job[pj];
    p_end = (pj + 1 < p.njobs) ? p.job[pj + 1].tile0 : p.ntiles;
    const int64_t sb = J.stride * C::ESZ;
    const int64_t row0 = (int64_t)(it - J.tile0) * C::RW;
    i_left = J.rows - row0;
    i_step = C::RW * sb;
    i_qstep = C::RPQ * sb;
    i_src = reinterpret_cast<const uint8_t*>(J.x) + (row0 + lane_cr) * sb + (lane % C::CPR) * 16;
  };
  set_issue_job();
  auto issue = [&](int stg) {
    if (it < t_end) {
      if (it >= p_end) {  // a warp's tiles only move forward
        while (it >= p_end) { ++pj; p_end = (pj + 1 < p.njobs) ? p.job[pj + 1].tile0 : p.ntiles; }
        set_issue_job();
      }
      uint8_t* dst = in_dst + stg * IT::BYTES;
      if (i_left >= C::RW) {
#pragma unroll
        for (int q = 0; q < C::CHUNKS; ++q) cp_async16(dst + q * C::RPQ * IT::STRIDE, i_src + q * i_qstep, 16);
      } else {  // the job's last tile: rows past its end are zero-filled
        const uint8_t* x0 = reinterpret_cast<const uint8_t*>(p.job[pj].x);
#pragma unroll
        for (int q = 0; q < C::CHUNKS; ++q) {
          const bool ok = q * C::RPQ + lane_cr < i_left;
          cp_async16(dst + q * C::RPQ * IT::STRIDE, ok ? i_src + q * i_qstep : x0, ok ? 16 : 0);
        }
      }
      i_src += i_step;
      i_left -= C::RW;
      ++it;
    }
    cp_async_commit();
  };
#pragma unroll
  for (int s = 0; s < kNS - 1; ++s) issue(s);

  // ---- compute cursor ----
  WarpJob* wj = reinterpret_cast<WarpJob*>(wsm + C::W_JOB);
  int c_end = t;                 // first tile after the current job (forces a job load)
  int64_t c_row0 = 0;            // the tile's first row within its job
  int64_t c_left = 0;            // rows of the job from c_row0
  bool c_dense = true;
  // copy-out: this lane's 16-byte chunk(s) of the current tile and the bytes
  // between consecutive tiles of its plane
  uint8_t* o_dst[C::ROUNDS];
  int o_step[C::ROUNDS];
#pragma unroll
  for (int q = 0; q < C::ROUNDS; ++q) { o_dst[q] = nullptr; o_step[q] = 0; }
  uint2 msk[8];
#pragma unroll
  for (int m = 0; m < 8; ++m) msk[m] = make_uint2(0u, 0u);
  // re-decision queue: qn entries (warp-uniform), moved to the launch's queue
  // in global memory when fewer than one tile's worst case of free entries is
  // left, and at the end
  using QG = QGeo<D>;
  uint4* const qb = reinterpret_cast<uint4*>(wsm + C::W_Q);
  int qn = 0;
  constexpr int q_hi = kQ - QG::kMaxPerTile;

  static_assert((kNS & (kNS - 1)) == 0, "stage ring size");
  int stage = 0;
  // Iterations ahead that need no checks: the computed tile is a full tile of
  // the current (dense) job and the prefetched tile a full tile of the issue
  // job inside the warp's range.  Set by the general iterations.
  int fast = 0;
  const float2* const etl = etab + (lane % C::TABR);
  while (t < t_end) {
    if (fast > 0) {
      // A stretch of `fast` tiles, each a full tile of the current dense job
      // whose prefetch is a full tile of the issue job: no per-tile checks, the
      // cursors are settled once after it.
      const int t_start = t, t_stop = t + fast;
      for (; t < t_stop; ++t) {
        if (qn > q_hi) break;   // the general iteration moves the queue first
        cp_async_wait<kNS - 2>();   // this warp tile has landed
        __syncwarp();               // ... and every lane is done with the previous one
        uint8_t* dst = in_dst + ((stage + kNS - 1) & (kNS - 1)) * IT::BYTES;
#pragma unroll
        for (int q = 0; q < C::CHUNKS; ++q) cp_async16(dst + q * C::RPQ * IT::STRIDE, i_src + q * i_qstep, 16);
        cp_async_commit();
        i_src += i_step;
        tile_body<D, TIn, N, B, MODE>(wsm + C::W_IN + stage * IT::BYTES, wsm, etl, C::RW, lane, msk, qb, qn, t, p);
        __syncwarp();
#pragma unroll
        for (int q = 0; q < C::ROUNDS; ++q) {
          const int ch = q * 32 + lane;
          if (ch < C::NCH)
            *reinterpret_cast<uint4*>(o_dst[q]) = *reinterpret_cast<const uint4*>(wsm + C::W_ANG + 16 * ch);
          o_dst[q] += o_step[q];
        }
        stage = (stage + 1) & (kNS - 1);
      }
      const int done = t - t_start;
      const int64_t adv = (int64_t)done * C::RW;
      c_row0 += adv;
      c_left -= adv;
      i_left -= adv;
      it += done;
      fast = 0;
      continue;
    }

    // ---- general tile: a job's first tile, tails, scattered slots, range ends,
    // and the queue's moves to global memory ----
    if (qn > q_hi) {
      spill_queue<D>(p, qb, qn, lane);
      qn = 0;
    }
    cp_async_wait<kNS - 2>();
    __syncwarp();
    issue((stage + kNS - 1) & (kNS - 1));
    if (t >= c_end) {  // next job
      const int cj = find_job(p, t);
      const EncJob& J = p.job[cj];
      c_end = (cj + 1 < p.njobs) ? p.job[cj + 1].tile0 : p.ntiles;
      const int rel = t - J.tile0;
      c_row0 = (int64_t)rel * C::RW;
      c_left = J.rows - c_row0;
      c_dense = J.slot == nullptr;
#pragma unroll
      for (int q = 0; q < C::ROUNDS; ++q) {
        const int ch = q * 32 + lane;
        if (ch < C::NA) { o_dst[q] = J.codes + 16 * ch; o_step[q] = C::RW * C::AB; }
        else if (ch < C::NA + C::NN) { o_dst[q] = J.norms + 16 * (ch - C::NA); o_step[q] = C::RW * C::NB; }
        else { o_dst[q] = J.hdr + 16 * (ch - C::NA - C::NN); o_step[q] = C::RW * C::HB; }
        o_dst[q] += (int64_t)rel * o_step[q];
      }
      if (lane == 0) {
        wj->codes = J.codes; wj->norms = J.norms; wj->hdr = J.hdr; wj->slot = J.slot; wj->capacity = J.capacity;
        wj->job = cj;
#pragma unroll
        for (int q = 0; q < 4; ++q) wj->signs[q] = J.signs[q];
      }
      const int l = lane % C::L;
#pragma unroll
      for (int m = 0; m < 8; ++m) {
        msk[m] = pair_sign_mask<C::ESZ>(J.signs, slot_pair<D>(l + C::L * m));
        if constexpr (C::ESZ == 2) msk[m].y = msk[m].x << 16;
      }
      __syncwarp();
    }
    const int nrows = c_left >= C::RW ? C::RW : (int)c_left;
    tile_body<D, TIn, N, B, MODE>(wsm + C::W_IN + stage * IT::BYTES, wsm, etl, nrows, lane, msk, qb, qn, t, p);
    __syncwarp();
    if (c_dense && nrows == C::RW) {
#pragma unroll
      for (int q = 0; q < C::ROUNDS; ++q) {
        const int ch = q * 32 + lane;
        if (ch < C::NCH)
          *reinterpret_cast<uint4*>(o_dst[q]) = *reinterpret_cast<const uint4*>(wsm + C::W_ANG + 16 * ch);
      }
    } else {
      copy_out_slow<C::AB, C::NB, C::HB>(wj, wsm + C::W_ANG, wsm + C::W_NRM, wsm + C::W_HDR, c_row0, nrows, lane);
    }
#pragma unroll
    for (int q = 0; q < C::ROUNDS; ++q) o_dst[q] += o_step[q];
    c_row0 += C::RW;
    c_left -= C::RW;
    stage = (stage + 1) & (kNS - 1);
    ++t;
    // c_left now counts the rows of the compute job from tile t, i_left those
    // of the issue job from tile it (the next to prefetch).
    const int64_t cf = c_dense ? c_left / C::RW : 0;
    const int64_t pf = min(min((int64_t)(p_end - it), i_left / C::RW), (int64_t)(t_end - it));
    const int64_t f = min(cf, pf);
    fast = f > 0 ? (int)f : 0;
  }
  if (qn > 0) spill_queue<D>(p, qb, qn, lane);
  cp_async_wait<0>();
}

// ---------------------------------------------------------------------------
// Fix-up of one encode launch (same stream, after it): the queue's entries,
// kFixChunk to a warp (the second look, then the exact path for the codes it
// leaves), then the rows whose entries found the queue full, each re-decided
// whole.  Grid-stride over both, so any grid size covers them.  The work is
// latency-bound (a warp takes its chunk's exact rows one after another), so
// the chunks are short and the grid wide.
// ---------------------------------------------------------------------------
constexpr int kFixWarps = 4;
constexpr int kFixChunk = 8;

template <int D, typename TIn, int N, int B, int MODE>
__global__ void __launch_bounds__(32 * kFixWarps) encode_fixup_kernel(const __grid_constant__ FixParams p) {
  constexpr int P = Geo<D>::P, RW = Geo<D>::RW;
  __shared__ long long scratch[kFixWarps][2 * P];
  __shared__ uint4 whole[kFixWarps][2];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long GW = (long long)gridDim.x * kFixWarps, gw = (long long)blockIdx.x * kFixWarps + warp;
  const unsigned long long appended = *p.gq_n;
  const long long n = (long long)min(appended, (unsigned long long)p.gq_cap);
  for (long long c = gw; kFixChunk * c < n; c += GW)
    flush_queue<D, TIn, N, B, MODE>(p.job, p.gq + 2 * kFixChunk * c, (int)min((long long)kFixChunk, n - kFixChunk * c),
                                    scratch[warp], lane);
  if (appended <= (unsigned long long)p.gq_cap) return;
  const long long nwords = ((long long)p.ntiles * RW + 31) / 32;
  for (long long w0 = gw * 32; w0 < nwords; w0 += GW * 32) {
    const long long wi = w0 + lane;
    const uint32_t word = wi < nwords ? p.ovf[wi] : 0u;
    unsigned live = __ballot_sync(0xffffffffu, word != 0u);
    while (live != 0u) {
      const int src = __ffs(live) - 1;
      live &= live - 1u;
      uint32_t bits = __shfl_sync(0xffffffffu, word, src);
      while (bits != 0u) {
        const int b = __ffs(bits) - 1;
        bits &= bits - 1u;
        const long long bit = (w0 + src) * 32 + b;
        const int j = find_job(p, (int)(bit / RW));
        const long long row = bit - (long long)p.job[j].tile0 * RW;
        if (row >= p.job[j].rows) continue;
        __syncwarp();
        if (lane == 0) {
          whole[warp][0] = make_uint4((uint32_t)j | (2u << 14), (uint32_t)row, 0u, 0u);
          whole[warp][1] = make_uint4(0u, 0u, 0u, 0u);
        }
        __syncwarp();
        flush_queue<D, TIn, N, B, MODE>(p.job, whole[warp], 1, scratch[warp], lane);
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Host-side launch helpers (called from tac_api.cu).
// ---------------------------------------------------------------------------
// phase: bit 0 launches the encode kernel, bit 1 its fix-up (3: both, in order).
template <int D, typename TIn, int N, int B, int MODE>
static cudaError_t launch_encode_v(const EncParams& p, int grid_cap, cudaStream_t st, int phase) {
  using C = Enc<D, TIn, N, B, MODE>;
  auto kern = encode_kernel<D, TIn, N, B, MODE>;
  static std::atomic<int> configured[64];   // per device; concurrent first calls set the same
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && configured[dev].load(std::memory_order_acquire) == 0) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    configured[dev].store(1, std::memory_order_release);
  }
  // resident CTAs per SM of both kernels, found once per device
  static std::atomic<int> occ[64][2];
  int per_sm = dev >= 0 && dev < 64 ? occ[dev][0].load(std::memory_order_acquire) : 0;
  int fix_sm = dev >= 0 && dev < 64 ? occ[dev][1].load(std::memory_order_acquire) : 0;
  auto fix = encode_fixup_kernel<D, TIn, N, B, MODE>;
  if (per_sm == 0 || fix_sm == 0) {
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kEncThreads, C::SMEM);
    if (e != cudaSuccess) return e;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&fix_sm, fix, 32 * kFixWarps, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    if (fix_sm < 1) fix_sm = 1;
    if (dev >= 0 && dev < 64) {
      occ[dev][0].store(per_sm, std::memory_order_release);
      occ[dev][1].store(fix_sm, std::memory_order_release);
    }
  }
  int grid = grid_cap * per_sm;
  const int need = (p.ntiles + kEncWarps - 1) / kEncWarps;
  if (grid > need) grid = need;
  if (grid < 1) return cudaSuccess;   // no rows: neither kernel runs
  if (phase & 1) {
    kern<<<grid, kEncThreads, C::SMEM, st>>>(p);
    const cudaError_t le = cudaGetLastError();
    if (le != cudaSuccess) return le;
  }
  if (!(phase & 2)) return cudaSuccess;
  // the fix-up: enough warps for the queue's capacity, up to a full GPU
  FixParams f;
  f.job = p.gjobs;
  f.gq = p.gq;
  f.gq_n = p.gq_n;
  f.ovf = p.ovf;
  f.gq_cap = p.gq_cap;
  f.njobs = p.njobs;
  f.ntiles = p.ntiles;
  const int64_t chunks = (p.gq_cap + kFixChunk - 1) / kFixChunk;
  int64_t fgrid = (int64_t)grid_cap * fix_sm;
  fgrid = std::min<int64_t>(fgrid, (chunks + kFixWarps - 1) / kFixWarps);
  if (fgrid < 1) fgrid = 1;
  fix<<<(int)fgrid, 32 * kFixWarps, 0, st>>>(f);
  return cudaGetLastError();
}

// One kernel per supported (n, norm bits, mode): n in {2, 4, ..., 256, 48, 56},
// (B, mode) in {(4, linear), (4, log), (8, linear), (8, log), (32, fp32)}.
template <int D, typename TIn>
static cudaError_t launch_encode_t(const EncParams& p, int n, int b, int mode, int sms, cudaStream_t st, int phase) {
#define TAC_ENC_N(NN)                                                                                   \
  if (n == NN) {                                                                                        \
    if (mode == TAC_NORM_FP32) return b == 32 ? launch_encode_v<D, TIn, NN, 32, TAC_NORM_FP32>(p, sms, st, phase) \
                                              : cudaErrorInvalidValue;                                  \
    if (b == 4) return mode == TAC_NORM_LOG ? launch_encode_v<D, TIn, NN, 4, TAC_NORM_LOG>(p, sms, st, phase)     \
                                            : launch_encode_v<D, TIn, NN, 4, TAC_NORM_LINEAR>(p, sms, st, phase); \
    if (b == 8) return mode == TAC_NORM_LOG ? launch_encode_v<D, TIn, NN, 8, TAC_NORM_LOG>(p, sms, st, phase)     \
                                            : launch_encode_v<D, TIn, NN, 8, TAC_NORM_LINEAR>(p, sms, st, phase); \
    return cudaErrorInvalidValue;                                                                       \
  }
  TAC_ENC_N(2) TAC_ENC_N(4) TAC_ENC_N(8) TAC_ENC_N(16) TAC_ENC_N(32) TAC_ENC_N(64) TAC_ENC_N(128)
  TAC_ENC_N(256) TAC_ENC_N(48) TAC_ENC_N(56)
#undef TAC_ENC_N
  return cudaErrorInvalidValue;
}

// Instances: the build compiles this file once per (d, dtype) with
// -DTAC_INST_D=<d> -DTAC_INST_BF16=1|-DTAC_INST_F32=1 so they compile in parallel;
// without those flags every instance is compiled here.
#if !defined(TAC_INST_D)
#define TAC_ALL_INSTANCES 1
#define TAC_INST_D 0
#endif
#ifndef TAC_INST_BF16
#define TAC_INST_BF16 0
#endif
#ifndef TAC_INST_F32
#define TAC_INST_F32 0
#endif
#define TAC_ENC_INSTANCE(DD, NAME, T)                                                                 \
  cudaError_t launch_encode_##DD##_##NAME(const EncParams& p, int n, int b, int mode, int sms,       \
                                          cudaStream_t st, int phase) {                              \
    return launch_encode_t<DD, T>(p, n, b, mode, sms, st, phase);                                    \
  }
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 16 && TAC_INST_BF16)
TAC_ENC_INSTANCE(16, bf16, __nv_bfloat16)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 32 && TAC_INST_BF16)
TAC_ENC_INSTANCE(32, bf16, __nv_bfloat16)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 64 && TAC_INST_BF16)
TAC_ENC_INSTANCE(64, bf16, __nv_bfloat16)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 128 && TAC_INST_BF16)
TAC_ENC_INSTANCE(128, bf16, __nv_bfloat16)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 16 && TAC_INST_F32)
TAC_ENC_INSTANCE(16, f32, float)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 32 && TAC_INST_F32)
TAC_ENC_INSTANCE(32, f32, float)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 64 && TAC_INST_F32)
TAC_ENC_INSTANCE(64, f32, float)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 128 && TAC_INST_F32)
TAC_ENC_INSTANCE(128, f32, float)
#endif
#undef TAC_ENC_INSTANCE

}  // namespace tac
