// TurboAngle encode kernel for sm_103a (Alg. 1 + Sec. 3.3 / Eq. 2 of arXiv 2603.27467).
//
// One thread owns one head vector (row) of a 128-row tile:
//   1. the tile is staged global -> shared with cp.async (coalesced 16-byte
//      chunks, double buffered, XOR-swizzled rows so per-row reads are
//      bank-conflict free);
//   2. D (sign XOR on the raw bits) and the unnormalized Walsh-Hadamard butterfly
//      run in registers on packed fp32 pairs (FADD2/FFMA2).  The element-pair
//      stage (input bit 0) is never executed: for output pair i the butterfly
//      halves E_i = WHT_i(x_even), O_i = WHT_i(x_odd) give
//      (y_2i, y_2i+1) = (E_i + O_i, E_i - O_i), so r_i^2 = 2 (E_i^2 + O_i^2) / d
//      (normalized) and the angle test is done directly on (E_i, O_i);
//   3. Alg. 1's k_i = floor(n theta/2pi + 1/2) mod n is decided by an exact
//      geometric test: a candidate edge e = floor(n theta~/2pi) from an fp32
//      atan2, then the sign of the cross product of (E, O) with the edge
//      direction.  The test is certified by a rigorous fp32 error bound (the
//      butterfly's rounding plus the product's); pairs inside the bound are
//      re-decided by the warp in fp64 from the staged input (exact sums);
//   4. Eq. 2 norm codes (linear, or log-space) against the stored fp32 (r_min, r_max);
//   5. LSB-first packing in registers, records staged in shared memory and
//      written with coalesced 16-byte stores (or to per-row slots: scatter-append).
#include "tac_common.cuh"

namespace tac {

template <int D, typename TIn>
struct Enc {
  static constexpr int P = D / 2;
  static constexpr int ESZ = (int)sizeof(TIn);
  static constexpr int ROWB = D * ESZ;             // staged input row bytes
  static constexpr int CPR = ROWB / 16;            // 16-byte chunks per row
  static constexpr int IN_B = kTileRows * ROWB;    // one input buffer
  static constexpr int ABMAX = P;                  // angle record bytes at w = 8
  static constexpr int NBMAX = P;                  // norm record bytes at b = 8
  static constexpr int LOGD = (D == 16) ? 4 : (D == 32) ? 5 : (D == 64) ? 6 : 7;
  // shared memory layout (bytes)
  static constexpr int OFF_IN = 0;
  static constexpr int OFF_ANG = OFF_IN + 2 * IN_B;
  static constexpr int OFF_NRM = OFF_ANG + kTileRows * ABMAX;
  static constexpr int OFF_HDR = OFF_NRM + kTileRows * NBMAX;
  static constexpr int OFF_TAB = OFF_HDR + kTileRows * 8;
  static constexpr int OFF_MSK = OFF_TAB + kTabEntries * 8;
  static constexpr int SMEM = OFF_MSK + P * 8;
};

// Store NW little-endian words (a packed record) to shared memory, with the
// widest vector the record stride allows.
template <int BYTES>
__device__ __forceinline__ void stage_record(uint8_t* dst, const uint32_t* w) {
  if constexpr (BYTES % 16 == 0) {
#pragma unroll
    for (int q = 0; q < BYTES / 16; ++q)
      reinterpret_cast<uint4*>(dst)[q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
  } else if constexpr (BYTES % 8 == 0) {
#pragma unroll
    for (int q = 0; q < BYTES / 8; ++q) reinterpret_cast<uint2*>(dst)[q] = make_uint2(w[2 * q], w[2 * q + 1]);
  } else if constexpr (BYTES % 4 == 0) {
#pragma unroll
    for (int q = 0; q < BYTES / 4; ++q) reinterpret_cast<uint32_t*>(dst)[q] = w[q];
  } else {
#pragma unroll
    for (int q = 0; q < BYTES; ++q) dst[q] = (uint8_t)(w[q >> 2] >> (8 * (q & 3)));
  }
}

// Copy `bytes` bytes shared -> global with the whole CTA (16-byte stores when both
// sides allow it; both bases are 16-byte aligned by construction).
__device__ __forceinline__ void cta_copy_out(uint8_t* g, const uint8_t* s, int bytes, int tid) {
  const int n16 = bytes >> 4;
  for (int q = tid; q < n16; q += kThreads)
    reinterpret_cast<uint4*>(g)[q] = reinterpret_cast<const uint4*>(s)[q];
  for (int q = (n16 << 4) + tid; q < bytes; q += kThreads) g[q] = s[q];
}

// Copy one record of BYTES bytes from shared memory to a global slot.
template <int BYTES>
__device__ __forceinline__ void copy_record(uint8_t* g, const uint8_t* s) {
  if constexpr (BYTES % 16 == 0) {
#pragma unroll
    for (int q = 0; q < BYTES / 16; ++q) reinterpret_cast<uint4*>(g)[q] = reinterpret_cast<const uint4*>(s)[q];
  } else if constexpr (BYTES % 8 == 0) {
#pragma unroll
    for (int q = 0; q < BYTES / 8; ++q) reinterpret_cast<uint2*>(g)[q] = reinterpret_cast<const uint2*>(s)[q];
  } else if constexpr (BYTES % 4 == 0) {
#pragma unroll
    for (int q = 0; q < BYTES / 4; ++q) reinterpret_cast<uint32_t*>(g)[q] = reinterpret_cast<const uint32_t*>(s)[q];
  } else {
#pragma unroll
    for (int q = 0; q < BYTES; ++q) g[q] = s[q];
  }
}

// Issue the cp.async copies of tile `t` (rows [row0, row0 + 128) of job j) into `buf`.
template <int D, typename TIn>
__device__ __forceinline__ void issue_tile_load(const EncJob& J, int row0, uint8_t* buf, int tid) {
  using C = Enc<D, TIn>;
  const uint8_t* x = reinterpret_cast<const uint8_t*>(J.x);
  const int64_t rows = J.rows;
#pragma unroll 4
  for (int q = 0; q < C::CPR; ++q) {
    const int id = q * kThreads + tid;
    const int r = id / C::CPR;
    const int c = id - r * C::CPR;
    const int64_t grow = (int64_t)row0 + r;
    const bool ok = grow < rows;
    const uint8_t* src = ok ? x + (grow * J.stride) * C::ESZ + c * 16 : x;
    uint8_t* dst = buf + r * C::ROWB + ((c ^ row_swz<C::ROWB>(r)) << 4);
    cp_async16(dst, src, ok ? 16 : 0);
  }
}

// Sign masks for the staged element pairs: for pair i, XOR words that flip the
// IEEE sign bit of x_2i and x_2i+1 where s_j = -1 (D of Sec. 2).
template <int D, typename TIn>
__device__ __forceinline__ void build_masks(const EncJob& J, uint2* msk, int tid) {
  using C = Enc<D, TIn>;
  for (int i = tid; i < C::P; i += kThreads) {
    const uint32_t b0 = (J.signs[(2 * i) >> 5] >> ((2 * i) & 31)) & 1u;
    const uint32_t b1 = (J.signs[(2 * i + 1) >> 5] >> ((2 * i + 1) & 31)) & 1u;
    if constexpr (C::ESZ == 2) msk[i] = make_uint2((b0 << 15) | (b1 << 31), 0u);
    else msk[i] = make_uint2(b0 << 31, b1 << 31);
  }
}

// Exact re-decision of pair i of tile row rr by one warp (all lanes call it with
// the same arguments).  E_i, O_i are summed in fp64 from the staged input (each
// term is an exactly representable signed input element), the candidate edge is
// taken from an fp32 atan2 of the exact values and the edge test is evaluated in
// fp64 against an fp64 edge direction.  Returns k (valid in every lane).
template <int D, typename TIn>
__device__ __noinline__ int exact_angle_code(const EncJob& J, const uint8_t* in, int rr, int i, int lane) {
  using C = Enc<D, TIn>;
  const int n = 1 << J.w;
  double Ep = 0.0, Op = 0.0;
  const uint8_t* row = in + rr * C::ROWB;
  const int sw = row_swz<C::ROWB>(rr);
  for (int jj = lane; jj < C::P; jj += 32) {
    const int j0 = 2 * jj, j1 = 2 * jj + 1;
    float x0, x1;
    if constexpr (C::ESZ == 2) {
      const int c = (j0 * 2) >> 4, o = (j0 * 2) & 15;
      const uint32_t w = *reinterpret_cast<const uint32_t*>(row + ((c ^ sw) << 4) + o);
      x0 = bf16lo(w); x1 = bf16hi(w);
    } else {
      const int c = (j0 * 4) >> 4, o = (j0 * 4) & 15;
      const float2 w = *reinterpret_cast<const float2*>(row + ((c ^ sw) << 4) + o);
      x0 = w.x; x1 = w.y;
    }
    if ((J.signs[j0 >> 5] >> (j0 & 31)) & 1u) x0 = -x0;
    if ((J.signs[j1 >> 5] >> (j1 & 31)) & 1u) x1 = -x1;
    const bool neg = __popc((unsigned)(i & jj)) & 1;
    Ep += neg ? -(double)x0 : (double)x0;
    Op += neg ? -(double)x1 : (double)x1;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    Ep += __shfl_xor_sync(0xffffffffu, Ep, off);
    Op += __shfl_xor_sync(0xffffffffu, Op, off);
  }
  if (Ep == 0.0 && Op == 0.0) return 0;  // pair (0, 0) -> bin 0
  const float th = atan2f((float)(Ep - Op), (float)(Ep + Op));
  const int e = ((int)floorf(th * ((float)n * 0.15915494309189535f))) & (n - 1);
  const double2 ab = cos_sin_q8_d(edge_q8(e, n), n);
  const double m = fma(Ep, ab.x, -(Op * ab.y));
  return (e + (m >= 0.0 ? 1 : 0)) & (n - 1);
}

// Encode this thread's row (tile row `tr`) of the staged tile; W = log2 n, B = norm bits.
template <int D, typename TIn, int W, int B>
__device__ __forceinline__ void encode_row(const EncJob& J, float2 (&v)[D / 2], uint8_t* smem,
                                           const float2* etab, int tr, bool live,
                                           uint64_t& flagmask) {
  using C = Enc<D, TIn>;
  constexpr int P = C::P;
  constexpr int n = 1 << W;
  constexpr int AB = P * W / 8;   // angle record bytes
  constexpr int NB = P * B / 8;   // norm record bytes
  constexpr int AW = (P * W + 31) / 32;
  constexpr int NW = (P * B + 31) / 32;
  constexpr int L = (1 << B) - 1;
  const float k2 = 2.0f / (float)D;

  // Pass 1: pair energies s_i = E_i^2 + O_i^2 (r_i^2 = 2 s_i / d), their sum and range.
  float S = 0.f, smin = __int_as_float(0x7f800000), smax = 0.f;
#pragma unroll
  for (int i = 0; i < P; ++i) {
    const float s = __fmaf_rn(v[i].x, v[i].x, __fmul_rn(v[i].y, v[i].y));
    S = __fadd_rn(S, s);
    smin = fminf(smin, s);
    smax = fmaxf(smax, s);
  }

  // Stored header (Sec. 3.3: fp32 min and max of the pair norms).
  float hmin, hmax, qscale, qbase, sfloor = 0.f;
  if (J.mode == TAC_NORM_LINEAR) {
    hmin = __fsqrt_rn(smin * k2);
    hmax = __fsqrt_rn(smax * k2);
    qscale = (hmax > hmin) ? __fdiv_rn((float)L, __fsub_rn(hmax, hmin)) : 0.f;
    qbase = hmin;
  } else {  // log-space: norms floored at 2^-24 r_max
    sfloor = smax * 3.5527136788005009e-15f;  // 2^-48 on the energy = 2^-24 on the norm
    hmin = __fsqrt_rn(fmaxf(smin, sfloor) * k2);
    hmax = __fsqrt_rn(smax * k2);
    const float lmin = log2f(hmin), lmax = log2f(hmax);
    qscale = (hmax > hmin && lmax > lmin) ? __fdiv_rn((float)L, __fsub_rn(lmax, lmin)) : 0.f;
    qbase = lmin;
  }

  // Certification bound for the edge test: the butterfly's rounding gives
  // |dE|, |dO| <= (log2 d - 1) u ||x||_1 (first order) with ||x||_1 <= sqrt(d) ||x||_2
  // = sqrt(2 S); the edge direction (<= 1 ulp each component), the product and the
  // fma add <= 4 u (|E| + |O|) <= 4 u sqrt(2 smax).  5 u and the 1.002 factor cover
  // the rounding of S, smax and of the bound itself.
  const float tau = 1.002f * kU * ((float)(C::LOGD - 1) * sqrtf(2.f * S) + 5.f * sqrtf(2.f * smax));
  // Pairs whose norm is so small that the fp32 angle may be off by a quarter bin
  // are re-decided too: r_EO < 4 n tau_y / pi.
  const float ty = (float)(C::LOGD - 1) * kU * sqrtf(2.f * S) * 1.002f;
  const float rthr = ty * (4.f * (float)n / 3.14159265f);
  const float sthr = rthr * rthr;

  uint32_t aw[AW], nw[NW];
#pragma unroll
  for (int q = 0; q < AW; ++q) aw[q] = 0u;
#pragma unroll
  for (int q = 0; q < NW; ++q) nw[q] = 0u;

  const float nscale = (float)n * 0.15915494309189535f;  // n / (2 pi)
  const float2* et = etab + tab_offset(W);
  uint64_t fm = 0;

#pragma unroll
  for (int i = 0; i < P; ++i) {
    const float E = v[i].x, O = v[i].y;
    const float s = __fmaf_rn(E, E, __fmul_rn(O, O));
    // --- angle code (Alg. 1) ---
    const float th = atan2f(__fsub_rn(E, O), __fadd_rn(E, O));
    const int e = __float2int_rd(th * nscale) & (n - 1);
    const float2 ab = et[e];
    const float m = __fmaf_rn(E, ab.x, -__fmul_rn(O, ab.y));
    int k = (e + (m >= 0.f ? 1 : 0)) & (n - 1);
    if (E == 0.f && O == 0.f) k = 0;
    if (fabsf(m) < tau || s < sthr) fm |= (1ull << i);
    // --- norm code (Eq. 2) ---
    float val;
    if (J.mode == TAC_NORM_LINEAR) val = __fsqrt_rn(s * k2);
    else val = 0.5f * log2f(fmaxf(s, sfloor) * k2);
    int c = __float2int_rd(__fmaf_rn(__fsub_rn(val, qbase), qscale, 0.5f));
    c = min(max(c, 0), L);
    // --- pack (LSB-first) ---
    {
      const int bit = i * W;
      const int wi = bit >> 5, sh = bit & 31;
      aw[wi] |= (uint32_t)k << sh;
      if (sh + W > 32) aw[wi + 1] |= (uint32_t)k >> (32 - sh);
    }
    {
      const int bit = i * B;
      nw[bit >> 5] |= (uint32_t)c << (bit & 31);
    }
  }
  flagmask = live ? fm : 0ull;

  if (live) {
    stage_record<AB>(smem + C::OFF_ANG + tr * AB, aw);
    stage_record<NB>(smem + C::OFF_NRM + tr * NB, nw);
    reinterpret_cast<float2*>(smem + C::OFF_HDR)[tr] = make_float2(hmin, hmax);
  }
}

template <int D, typename TIn, int W, int B>
__device__ __forceinline__ void copy_tile_out(const EncJob& J, const uint8_t* smem, int row0, int nrows,
                                              int tid) {
  using C = Enc<D, TIn>;
  constexpr int P = C::P;
  constexpr int AB = P * W / 8;
  constexpr int NB = P * B / 8;
  if (J.slot == nullptr) {
    cta_copy_out(J.codes + (int64_t)row0 * AB, smem + C::OFF_ANG, nrows * AB, tid);
    cta_copy_out(J.norms + (int64_t)row0 * NB, smem + C::OFF_NRM, nrows * NB, tid);
    cta_copy_out(J.hdr + (int64_t)row0 * 8, smem + C::OFF_HDR, nrows * 8, tid);
  } else if (tid < nrows) {
    const int64_t s = J.slot[row0 + tid];
    if (s < 0 || s >= J.capacity) return;  // out-of-range slots are skipped
    copy_record<AB>(J.codes + s * AB, smem + C::OFF_ANG + tid * AB);
    copy_record<NB>(J.norms + s * NB, smem + C::OFF_NRM + tid * NB);
    reinterpret_cast<float2*>(J.hdr)[s] = reinterpret_cast<const float2*>(smem + C::OFF_HDR)[tid];
  }
}

// Patch code i (W bits) of the staged angle record of row rr.
__device__ __forceinline__ void patch_code(uint8_t* rec, int i, int W, int k) {
  for (int t = 0; t < W; ++t) {
    const int bit = i * W + t;
    const uint8_t mask = (uint8_t)(1u << (bit & 7));
    if ((k >> t) & 1) rec[bit >> 3] |= mask; else rec[bit >> 3] &= (uint8_t)~mask;
  }
}

template <int D, typename TIn, int W, int B>
__device__ __forceinline__ void tile_body(const EncJob& J, uint8_t* smem, const uint8_t* in, int row0,
                                          int nrows, int tid) {
  using C = Enc<D, TIn>;
  constexpr int P = C::P;
  const bool live = tid < nrows;
  const uint2* msk = reinterpret_cast<const uint2*>(smem + C::OFF_MSK);
  const float2* etab = reinterpret_cast<const float2*>(smem + C::OFF_TAB);

  // Load this thread's row from the swizzled tile, apply D, widen to fp32 pairs.
  float2 v[P];
  {
    const uint8_t* row = in + tid * C::ROWB;
    const int sw = row_swz<C::ROWB>(tid);
#pragma unroll
    for (int c = 0; c < C::CPR; ++c) {
      const uint4 q = *reinterpret_cast<const uint4*>(row + ((c ^ sw) << 4));
      const uint32_t wv[4] = {q.x, q.y, q.z, q.w};
      if constexpr (C::ESZ == 2) {
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int i = 4 * c + t;
          const uint32_t w = wv[t] ^ msk[i].x;
          v[i] = make_float2(bf16lo(w), bf16hi(w));
        }
      } else {
#pragma unroll
        for (int t = 0; t < 2; ++t) {
          const int i = 2 * c + t;
          v[i] = make_float2(__uint_as_float(wv[2 * t] ^ msk[i].x), __uint_as_float(wv[2 * t + 1] ^ msk[i].y));
        }
      }
    }
  }
  // Unnormalized Walsh-Hadamard butterfly over the pair index (input bits 1..log2 d - 1).
#pragma unroll
  for (int h = 1; h < P; h <<= 1) {
#pragma unroll
    for (int i = 0; i < P; ++i) {
      if ((i & h) == 0) {
        const float2 a = v[i], b = v[i + h];
        v[i] = add2(a, b);
        v[i + h] = sub2(a, b);
      }
    }
  }

  uint64_t fm = 0;
  encode_row<D, TIn, W, B>(J, v, smem, etab, tid, live, fm);
  __syncwarp();

  // Exact re-decision of the uncertified pairs, one warp per pair.
  const int lane = tid & 31;
  const int wrow0 = tid & ~31;
  unsigned ball = __ballot_sync(0xffffffffu, fm != 0ull);
  while (ball) {
    const int owner = __ffs(ball) - 1;
    ball &= ball - 1;
    uint64_t m = __shfl_sync(0xffffffffu, fm, owner);
    const int rr = wrow0 + owner;
    while (m) {
      const int i = __ffsll((long long)m) - 1;
      m &= m - 1;
      const int k = exact_angle_code<D, TIn>(J, in, rr, i, lane);
      if (lane == 0) patch_code(smem + C::OFF_ANG + rr * (P * W / 8), i, W, k);
    }
    __syncwarp();
  }
}

template <int D, typename TIn>
__global__ void __launch_bounds__(kThreads, 2) encode_kernel(const __grid_constant__ EncParams p) {
  using C = Enc<D, TIn>;
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x;
  const int G = gridDim.x;
  int t = blockIdx.x;
  if (t >= p.ntiles) return;

  // Edge tables for every n = 2..256.
  float2* etab = reinterpret_cast<float2*>(smem + C::OFF_TAB);
  for (int idx = tid; idx < kTabEntries - 2; idx += kThreads) {
    const int w = 31 - __clz(idx + 2);
    const int e = idx - tab_offset(w);
    etab[idx] = cos_sin_q8(edge_q8(e, 1 << w), 1 << w);
  }

  int jid = find_job(p, t);
  build_masks<D, TIn>(p.job[jid], reinterpret_cast<uint2*>(smem + C::OFF_MSK), tid);

  // Prologue: two tiles in flight.
  {
    const EncJob& J = p.job[jid];
    issue_tile_load<D, TIn>(J, (t - J.tile0) * kTileRows, smem + C::OFF_IN, tid);
    cp_async_commit();
    const int t1 = t + G;
    if (t1 < p.ntiles) {
      const EncJob& J1 = p.job[find_job(p, t1)];
      issue_tile_load<D, TIn>(J1, (t1 - J1.tile0) * kTileRows, smem + C::OFF_IN + C::IN_B, tid);
    }
    cp_async_commit();
  }

  int cur = 0;
  for (; t < p.ntiles; t += G) {
    cp_async_wait<1>();
    __syncthreads();
    const EncJob& J = p.job[jid];
    const int row0 = (t - J.tile0) * kTileRows;
    const int nrows = (int)min((int64_t)kTileRows, J.rows - row0);
    const uint8_t* in = smem + C::OFF_IN + cur * C::IN_B;

#define TAC_ENC_CASE(WW)                                                              \
  case WW:                                                                            \
    if (J.b == 8) tile_body<D, TIn, WW, 8>(J, smem, in, row0, nrows, tid);            \
    else tile_body<D, TIn, WW, 4>(J, smem, in, row0, nrows, tid);                     \
    break;
    switch (J.w) {
      TAC_ENC_CASE(1) TAC_ENC_CASE(2) TAC_ENC_CASE(3) TAC_ENC_CASE(4)
      TAC_ENC_CASE(5) TAC_ENC_CASE(6) TAC_ENC_CASE(7) TAC_ENC_CASE(8)
      default: break;
    }
#undef TAC_ENC_CASE
    __syncthreads();

#define TAC_OUT_CASE(WW)                                                              \
  case WW:                                                                            \
    if (J.b == 8) copy_tile_out<D, TIn, WW, 8>(J, smem, row0, nrows, tid);            \
    else copy_tile_out<D, TIn, WW, 4>(J, smem, row0, nrows, tid);                     \
    break;
    switch (J.w) {
      TAC_OUT_CASE(1) TAC_OUT_CASE(2) TAC_OUT_CASE(3) TAC_OUT_CASE(4)
      TAC_OUT_CASE(5) TAC_OUT_CASE(6) TAC_OUT_CASE(7) TAC_OUT_CASE(8)
      default: break;
    }
#undef TAC_OUT_CASE

    // Refill this buffer with tile t + 2G; prepare the sign masks of tile t + G.
    const int t2 = t + 2 * G;
    if (t2 < p.ntiles) {
      const EncJob& J2 = p.job[find_job(p, t2)];
      issue_tile_load<D, TIn>(J2, (t2 - J2.tile0) * kTileRows, smem + C::OFF_IN + cur * C::IN_B, tid);
    }
    cp_async_commit();
    if (t + G < p.ntiles) {
      jid = find_job(p, t + G);
      build_masks<D, TIn>(p.job[jid], reinterpret_cast<uint2*>(smem + C::OFF_MSK), tid);
    }
    cur ^= 1;
  }
  cp_async_wait<0>();
}

// ---------------------------------------------------------------------------
// Host-side launch helpers (called from tac_api.cu).
// ---------------------------------------------------------------------------
template <int D, typename TIn>
static cudaError_t launch_encode_t(const EncParams& p, int grid_cap, cudaStream_t st) {
  using C = Enc<D, TIn>;
  auto kern = encode_kernel<D, TIn>;
  static int configured[64] = {0};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    configured[dev] = 1;
  }
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, C::SMEM);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) per_sm = 1;
  int grid = grid_cap * per_sm;
  if (grid > p.ntiles) grid = p.ntiles;
  if (grid < 1) return cudaSuccess;
  kern<<<grid, kThreads, C::SMEM, st>>>(p);
  return cudaGetLastError();
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
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 16 && TAC_INST_BF16)
cudaError_t launch_encode_16_bf16(const EncParams& p, int sms, cudaStream_t st) {
  return launch_encode_t<16, __nv_bfloat16>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 32 && TAC_INST_BF16)
cudaError_t launch_encode_32_bf16(const EncParams& p, int sms, cudaStream_t st) {
  return launch_encode_t<32, __nv_bfloat16>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 64 && TAC_INST_BF16)
cudaError_t launch_encode_64_bf16(const EncParams& p, int sms, cudaStream_t st) {
  return launch_encode_t<64, __nv_bfloat16>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 128 && TAC_INST_BF16)
cudaError_t launch_encode_128_bf16(const EncParams& p, int sms, cudaStream_t st) {
  return launch_encode_t<128, __nv_bfloat16>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 16 && TAC_INST_F32)
cudaError_t launch_encode_16_f32(const EncParams& p, int sms, cudaStream_t st) {
  return launch_encode_t<16, float>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 32 && TAC_INST_F32)
cudaError_t launch_encode_32_f32(const EncParams& p, int sms, cudaStream_t st) {
  return launch_encode_t<32, float>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 64 && TAC_INST_F32)
cudaError_t launch_encode_64_f32(const EncParams& p, int sms, cudaStream_t st) {
  return launch_encode_t<64, float>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 128 && TAC_INST_F32)
cudaError_t launch_encode_128_f32(const EncParams& p, int sms, cudaStream_t st) {
  return launch_encode_t<128, float>(p, sms, st);
}
#endif

}  // namespace tac
