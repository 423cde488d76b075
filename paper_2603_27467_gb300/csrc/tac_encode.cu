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
//      product of (E, O) with the edge direction.  The test is
//      certified by a rigorous bound on the fp32 error; the pairs it does not
//      certify (about 1e-4 of them) are re-decided by the warp from fp64 sums
//      of the staged input;
//   4. Eq. 2 norm codes (linear, or on log2 r) against the stored fp32 (r_min, r_max);
//   5. each lane packs its 8 codes LSB-first; the warp stages its records in
//      shared memory and writes them with one 16-byte store per lane (contiguous
//      slots) or per row (scatter-append slots).
#include "tac_common.cuh"

namespace tac {

// Edge directions (cos psi_e, sin psi_e) for every supported n in fp64, read
// warp-uniformly by the exact path.
namespace cx {
struct DEdgeTable { CS v[kTabEntries]; };
constexpr DEdgeTable make_d_edge_table() {
  DEdgeTable t{};
  for (int idx = 0; idx < kTabEntries; ++idx) {
    const int n = tab_n_of(idx), e = idx - tab_offset_n(n);
    t.v[idx] = cos_sin_q8(8 * e + 4 + n, n);
  }
  return t;
}
}  // namespace cx
__constant__ cx::DEdgeTable g_edge_d = cx::make_d_edge_table();

constexpr int kNS = 4;  // pipeline stages per warp: kNS - 1 warp tiles in flight
// CTA shape of the encode: 10 warps, two CTAs per SM (20 warps, up to 102
// registers a thread): the encode is issue-bound, and the extra warps hide
// more latency than the 128-register build's longer chains (3 % faster; 12
// warps at 80 registers emit more instructions).
constexpr int kEncWarps = 10;
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
  static constexpr int WARP_B = W_JOB + 64;
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

// Exact re-decision of pair i of warp-tile row rr by the whole warp (all lanes
// call it with the same arguments); returns k in every lane.  E_i = sum_j
// +-x_2j and O_i = sum_j +-x_2j+1 (each term an exactly representable signed
// input element) are summed in fp64 across the warp: relative error at most
// (P - 1) 2^-53 of ||x||_1, far inside the 1e-5 rad band the angle parity
// tolerates (the FP64 pipe is slow, but this path takes about 1e-4 of the
// pairs).  The candidate edge comes from the fp32 polynomial on the sums
// rounded to fp32 (scaled by a power of two when tiny, so that the reciprocal
// sees a normal number); the edge test m = E cos psi - O sin psi is evaluated
// in fp64 against the fp64 edge direction.
template <int D, typename TIn, int N>
__device__ __forceinline__ int exact_angle_code(const uint32_t* signs, const uint8_t* in, int rr, int i,
                                                int lane) {
  using G = Geo<D>;
  using IT = RowTile<D, (int)sizeof(TIn)>;
  constexpr int ESZ = (int)sizeof(TIn);
  constexpr int P = G::P;
  double e = 0.0, o = 0.0;
  const int ip = slot_pair<D>(i);   // the pair held in slot i
  const uint8_t* row = in + rr * IT::STRIDE;
#pragma unroll
  for (int j0 = 0; j0 < P; j0 += 32) {
    const int jj = j0 + lane;
    if (jj < P) {
      const int e0 = 2 * jj, e1 = 2 * jj + 1;
      float x0, x1;
      if constexpr (ESZ == 2) {
        const uint32_t u = *reinterpret_cast<const uint32_t*>(row + 4 * jj);
        x0 = bf16lo(u); x1 = bf16hi(u);
      } else {
        const float2 u = *reinterpret_cast<const float2*>(row + 8 * jj);
        x0 = u.x; x1 = u.y;
      }
      const bool neg = __popc((unsigned)(ip & jj)) & 1;
      if (((signs[e0 >> 5] >> (e0 & 31)) & 1u) != (uint32_t)neg) x0 = -x0;
      if (((signs[e1 >> 5] >> (e1 & 31)) & 1u) != (uint32_t)neg) x1 = -x1;
      e += (double)x0;
      o += (double)x1;
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    e += __shfl_xor_sync(0xffffffffu, e, off);
    o += __shfl_xor_sync(0xffffffffu, o, off);
  }
  if (e == 0.0 && o == 0.0) return 0;  // pair (0, 0) -> bin 0
  const double sc = (fabs(e) + fabs(o) < 1e-30) ? 18446744073709551616.0 : 1.0;   // exact 2^64
  const int ec = candidate_edge<N>((float)(e * sc), (float)(o * sc));
  const cx::CS dir = g_edge_d.v[tab_offset_n(N) + ec];
  const double m = fma(e, dir.c, -(o * dir.s));
  return wrap_bin<N>(ec + (m >= 0.0 ? 1 : 0));
}

// Patch code i (W bits) of a staged angle record (one lane).
template <int W>
__device__ __forceinline__ void patch_code(uint8_t* rec, int i, int k) {
  const int bit = i * W, b0 = bit >> 3, sh = bit & 7;
  const uint32_t mask = ((1u << W) - 1u) << sh;
  uint32_t v = rec[b0];
  if (sh + W > 8) v |= (uint32_t)rec[b0 + 1] << 8;
  v = (v & ~mask) | ((uint32_t)k << sh);
  rec[b0] = (uint8_t)v;
  if (sh + W > 8) rec[b0 + 1] = (uint8_t)(v >> 8);
}

// Encode this lane's 8 pairs of warp-tile row r (lane l of the row) and stage
// the records; N bins, B = norm bits, MODE = TAC_NORM_LINEAR / TAC_NORM_LOG /
// TAC_NORM_FP32 (B = 32: the pair norms themselves, no header).
template <int D, typename TIn, int N, int B, int MODE>
__device__ __forceinline__ void tile_body(const uint8_t* in, uint8_t* wsm, const float2* et, int nrows,
                                          int lane, const uint2 (&msk)[8], const uint32_t* signs) {
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
  const bool zero_row = !(smax > 0.f);

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
  float hmin = 0.f, hmax = 0.f, qs = 0.f, qo = 0.f, sfloor = 0.f;
  if constexpr (FP32N) {
    // no header: the norms are stored as they are (Sec. 3.1)
  } else if constexpr (MODE == TAC_NORM_LINEAR) {
    hmin = sqrt_approx(smin * k2);              // smin * sigma may still be subnormal
    hmax = (kEvenK2 ? rms * rk2 : sqrt_ftz(smax_s * k2)) * sr;
    const float sc = (float)Lq * rcp_approx(hmax - hmin);
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
    const float sc = (float)Lq * rcp_approx(lg2_ftz(hmax_s) - lmin_s);
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
  // (<= 1 ulp), the product and the fma add <= 4 u (|E| + |O|) <= 4 u sqrt(2 smax).
  const float rmx = rms * sr;
  const float ty = (float)(G::LOGD - 1) * kU * 1.01f * (sqrt_ftz(ssum * sigma) * sr);
  const float tau = ty + 5.f * kU * 1.4143f * rmx;
  // The per-pair norm functions below take s itself (pairs below the log floor
  // are clamped to it first), against the true-scale qs, qo: for inputs in the
  // supported range every nonzero s is a normal fp32 number, so the
  // flush-to-zero hardware forms see it unchanged.
  (void)qs; (void)qo; (void)sfloor;
  // Pairs whose norm is so small that the fp32 angle may be off by a quarter bin
  // are re-decided too: sqrt(s) < 4 n ty / pi.
  const float rthr = ty * (4.f * (float)n / 3.14159265f);
  const float sthr = rthr * rthr;

  // ---- pass 2: norm codes (Eq. 2), packing ----
  uint32_t nlo = 0, nhi = 0;
  float rn[FP32N ? 8 : 1];                      // fp32 norms r_j = sqrt(2 s_j / d)
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    // fields are disjoint and c <= Lq: the adds are ORs (one IMAD each)
    if constexpr (FP32N) {
      rn[j] = sqrt_approx(s[j] * k2);
    } else {
      float f;
      if constexpr (MODE == TAC_NORM_LINEAR) f = sqrt_ftz(s[j]);
      else f = lg2_ftz(fmaxf(s[j], sfloor));
      const uint32_t c = min(__float2uint_rd(__fmaf_rn(f, qs, qo)), (uint32_t)Lq);
      const int sn = j * B;
      if (sn < 32) nlo += c << sn; else nhi += c << (sn - 32);
    }
  }
  uint32_t fm = 0;
  if (zero_row) { alo = ahi = nlo = nhi = 0; hmin = hmax = 0.f; }
  else if (mmin < tau || lmin_s < sthr) {  // rare: name the uncertified pairs
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (am[j] < tau || s[j] < sthr) fm |= 1u << j;
  }
  if (!live) fm = 0;

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

  // ---- exact re-decision of the uncertified pairs, one warp per pair ----
  unsigned ball = __ballot_sync(0xffffffffu, fm != 0u);
  while (ball) {
    const int owner = __ffs(ball) - 1;
    ball &= ball - 1;
    uint32_t mm = __shfl_sync(0xffffffffu, fm, owner);
    const int rr = owner / L, ol = owner % L;
    while (mm) {
      const int j = __ffs(mm) - 1;
      mm &= mm - 1;
      const int i = 8 * ol + j;
      const int kk = exact_angle_code<D, TIn, N>(signs, in, rr, i, lane);
      if (lane == 0) patch_code<W>(wsm + C::W_ANG + rr * AB, i, kk);
    }
    __syncwarp();
  }
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
      const int t_stop = t + fast;
      for (; t < t_stop; ++t) {
        cp_async_wait<kNS - 2>();   // this warp tile has landed
        __syncwarp();               // ... and every lane is done with the previous one
        uint8_t* dst = in_dst + ((stage + kNS - 1) & (kNS - 1)) * IT::BYTES;
#pragma unroll
        for (int q = 0; q < C::CHUNKS; ++q) cp_async16(dst + q * C::RPQ * IT::STRIDE, i_src + q * i_qstep, 16);
        cp_async_commit();
        i_src += i_step;
        tile_body<D, TIn, N, B, MODE>(wsm + C::W_IN + stage * IT::BYTES, wsm, etl, C::RW, lane, msk, wj->signs);
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
      const int64_t adv = (int64_t)fast * C::RW;
      c_row0 += adv;
      c_left -= adv;
      i_left -= adv;
      it += fast;
      fast = 0;
      continue;
    }

    // ---- general tile: a job's first tile, tails, scattered slots, range ends ----
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
    tile_body<D, TIn, N, B, MODE>(wsm + C::W_IN + stage * IT::BYTES, wsm, etl, nrows, lane, msk, wj->signs);
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
  cp_async_wait<0>();
}

// ---------------------------------------------------------------------------
// Host-side launch helpers (called from tac_api.cu).
// ---------------------------------------------------------------------------
template <int D, typename TIn, int N, int B, int MODE>
static cudaError_t launch_encode_v(const EncParams& p, int grid_cap, cudaStream_t st) {
  using C = Enc<D, TIn, N, B, MODE>;
  auto kern = encode_kernel<D, TIn, N, B, MODE>;
  static int configured[64] = {0};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    configured[dev] = 1;
  }
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kEncThreads, C::SMEM);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) per_sm = 1;
  int grid = grid_cap * per_sm;
  const int need = (p.ntiles + kEncWarps - 1) / kEncWarps;
  if (grid > need) grid = need;
  if (grid < 1) return cudaSuccess;
  kern<<<grid, kEncThreads, C::SMEM, st>>>(p);
  return cudaGetLastError();
}

// One kernel per supported (n, norm bits, mode): n in {2, 4, ..., 256, 48, 56},
// (B, mode) in {(4, linear), (4, log), (8, linear), (8, log), (32, fp32)}.
template <int D, typename TIn>
static cudaError_t launch_encode_t(const EncParams& p, int n, int b, int mode, int sms, cudaStream_t st) {
#define TAC_ENC_N(NN)                                                                                   \
  if (n == NN) {                                                                                        \
    if (mode == TAC_NORM_FP32) return b == 32 ? launch_encode_v<D, TIn, NN, 32, TAC_NORM_FP32>(p, sms, st) \
                                              : cudaErrorInvalidValue;                                  \
    if (b == 4) return mode == TAC_NORM_LOG ? launch_encode_v<D, TIn, NN, 4, TAC_NORM_LOG>(p, sms, st)     \
                                            : launch_encode_v<D, TIn, NN, 4, TAC_NORM_LINEAR>(p, sms, st); \
    if (b == 8) return mode == TAC_NORM_LOG ? launch_encode_v<D, TIn, NN, 8, TAC_NORM_LOG>(p, sms, st)     \
                                            : launch_encode_v<D, TIn, NN, 8, TAC_NORM_LINEAR>(p, sms, st); \
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
                                          cudaStream_t st) {                                         \
    return launch_encode_t<DD, T>(p, n, b, mode, sms, st);                                           \
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
