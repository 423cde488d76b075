// TurboAngle encode kernel for sm_103a (Alg. 1 + Sec. 3.3 / Eq. 2 of arXiv 2603.27467).
//
// A 256-thread CTA encodes a tile of TR = 256/L rows; each row is shared by
// L = d/16 consecutive lanes and each lane owns 8 angle pairs (16 elements).
//   1. Tiles are staged global -> shared with cp.async (coalesced 16-byte
//      chunks, double buffered, padded rows).
//   2. D is a sign XOR on the raw input bits.  The unnormalized Walsh-Hadamard
//      butterfly runs in two register phases on packed fp32 pairs (FADD2/FFMA2):
//      phase A over the pair-index bits held in registers (lane l holds pairs
//      l + L*m), an intra-warp shared-memory transpose, phase B over the low
//      bits (lane l then holds pairs 8l..8l+7).  The element-pair stage (input
//      bit 0) is never executed: for output pair i the butterfly halves
//      E_i = WHT_i(x_even), O_i = WHT_i(x_odd) give (y_2i, y_2i+1) = (E+O, E-O),
//      so r_i^2 = 2 (E_i^2 + O_i^2) / d and the angle test works on (E_i, O_i).
//   3. Alg. 1's k_i = floor(n theta/2pi + 1/2) mod n is decided by an exact edge
//      test: a candidate edge from an octant-reduced arctangent polynomial
//      (max error 0.0038 rad: Rajan, Wang, Inkol, Joyal, "Efficient
//      approximations for the arctangent function", IEEE SPM 2006), then the sign
//      of the cross product of (E, O) with the edge direction.  The test is
//      certified by a rigorous bound on the fp32 error; pairs inside it are
//      re-decided by the warp in fp64 from the staged input (exact sums).
//   4. Eq. 2 norm codes (linear, or on log2 r) against the stored fp32 (r_min, r_max).
//   5. Each lane packs its 8 codes (8 log2(n) bits, 8 b bits) LSB-first; records
//      are staged in shared memory and written with coalesced stores, or to per-row
//      slots (scatter-append).
#include "tac_common.cuh"

namespace tac {

// fp64 edge directions (cos psi_e, sin psi_e) for every n = 2..256, read
// warp-uniformly by the exact-decision path.
__constant__ cx::EdgeTable g_edge_dir = cx::make_edge_table();

constexpr int kStages = 4;  // input tiles per CTA: 3 in flight while one is encoded

template <int D, typename TIn>
struct Enc {
  using G = Geo<D>;
  using IT = RowTile<D, (int)sizeof(TIn)>;
  static constexpr int P = G::P, L = G::L, TR = G::TR;
  static constexpr int ESZ = (int)sizeof(TIn);
  static constexpr int ABMAX = P;   // angle record bytes at w = 8
  static constexpr int NBMAX = P;   // norm record bytes at b = 8
  // shared memory layout (bytes)
  static constexpr int OFF_IN = 0;                           // kStages input tiles
  static constexpr int OFF_TP = OFF_IN + kStages * IT::BYTES; // transpose buffer
  static constexpr int OFF_ANG = OFF_TP + G::TP_B;           // staged angle records
  static constexpr int OFF_NRM = OFF_ANG + TR * ABMAX;       // staged norm records
  static constexpr int OFF_HDR = OFF_NRM + TR * NBMAX;       // staged headers
  static constexpr int OFF_TAB = OFF_HDR + TR * 8;           // edge tables, every n
  static constexpr int SMEM = OFF_TAB + kTabEntries * 8;
  static constexpr int CHUNKS = TR * IT::CPR / kThreads;     // cp.async chunks per thread
  static_assert(TR * IT::CPR % kThreads == 0, "tile chunks");
};

__device__ __forceinline__ void cta_copy_out(uint8_t* g, const uint8_t* s, int bytes, int tid) {
  const int n16 = bytes >> 4;
  for (int q = tid; q < n16; q += kThreads)
    reinterpret_cast<uint4*>(g)[q] = reinterpret_cast<const uint4*>(s)[q];
  for (int q = (n16 << 4) + tid; q < bytes; q += kThreads) g[q] = s[q];
}

// Copy BYTES bytes (one record) shared -> global at a slot.
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

// Store the low NBYTES bytes of v at a shared address aligned to gcd(NBYTES, 8).
template <int NBYTES>
__device__ __forceinline__ void store_bytes(uint8_t* dst, uint64_t v) {
  if constexpr (NBYTES == 8) {
    *reinterpret_cast<uint2*>(dst) = make_uint2((uint32_t)v, (uint32_t)(v >> 32));
  } else if constexpr (NBYTES == 4) {
    *reinterpret_cast<uint32_t*>(dst) = (uint32_t)v;
  } else if constexpr (NBYTES % 2 == 0) {
#pragma unroll
    for (int q = 0; q < NBYTES / 2; ++q) reinterpret_cast<uint16_t*>(dst)[q] = (uint16_t)(v >> (16 * q));
  } else {
#pragma unroll
    for (int q = 0; q < NBYTES; ++q) dst[q] = (uint8_t)(v >> (8 * q));
  }
}

template <int D, typename TIn>
__device__ __forceinline__ void issue_tile_load(const EncJob& J, int row0, uint8_t* buf, int tid) {
  using C = Enc<D, TIn>;
  using IT = typename C::IT;
  const uint8_t* x = reinterpret_cast<const uint8_t*>(J.x);
#pragma unroll
  for (int q = 0; q < C::CHUNKS; ++q) {
    const int id = q * kThreads + tid;
    const int r = id / IT::CPR;
    const int c = id - r * IT::CPR;
    const int64_t grow = (int64_t)row0 + r;
    const bool ok = grow < J.rows;
    const uint8_t* src = ok ? x + (grow * J.stride) * C::ESZ + c * 16 : x;
    cp_async16(buf + r * IT::STRIDE + c * 16, src, ok ? 16 : 0);
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
  using IT = typename C::IT;
  const int n = 1 << J.w;
  double Ep = 0.0, Op = 0.0;
  const uint8_t* row = in + rr * IT::STRIDE;
  for (int jj = lane; jj < C::P; jj += 32) {
    const int j0 = 2 * jj, j1 = 2 * jj + 1;
    float x0, x1;
    if constexpr (C::ESZ == 2) {
      const uint32_t w = *reinterpret_cast<const uint32_t*>(row + 4 * jj);
      x0 = bf16lo(w); x1 = bf16hi(w);
    } else {
      const float2 w = *reinterpret_cast<const float2*>(row + 8 * jj);
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
  const cx::CS ab = g_edge_dir.v[tab_offset(J.w) + e];
  const double m = fma(Ep, ab.c, -(Op * ab.s));
  return (e + (m >= 0.0 ? 1 : 0)) & (n - 1);
}

// Patch code i (W bits) of a staged angle record.
__device__ __forceinline__ void patch_code(uint8_t* rec, int i, int W, int k) {
  for (int t = 0; t < W; ++t) {
    const int bit = i * W + t;
    const uint8_t mask = (uint8_t)(1u << (bit & 7));
    if ((k >> t) & 1) rec[bit >> 3] |= mask; else rec[bit >> 3] &= (uint8_t)~mask;
  }
}

// Encode one tile: this thread's 8 pairs of row r (lane l) of the staged tile.
// W = log2 n, B = norm bits.
template <int D, typename TIn, int W, int B>
__device__ __forceinline__ void tile_body(const EncJob& J, uint8_t* smem, const uint8_t* in, int nrows,
                                          int tid, const uint2 (&msk)[8]) {
  using C = Enc<D, TIn>;
  using G = Geo<D>;
  using IT = typename C::IT;
  constexpr int P = C::P, L = C::L;
  constexpr int n = 1 << W;
  constexpr int AB = P * W / 8;           // angle record bytes
  constexpr int NB = P * B / 8;           // norm record bytes
  constexpr int Lq = (1 << B) - 1;
  const int r = tid / L, l = tid % L;
  const bool live = r < nrows;

  // ---- load 8 pairs (i = l + L*m), apply D, widen ----
  float2 v[8];
  {
    const uint8_t* row = in + r * IT::STRIDE;
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      const int i = l + L * m;
      if constexpr (C::ESZ == 2) {
        const uint32_t w = *reinterpret_cast<const uint32_t*>(row + 4 * i) ^ msk[m].x;
        v[m] = make_float2(bf16lo(w), bf16hi(w));
      } else {
        const uint2 w = *reinterpret_cast<const uint2*>(row + 8 * i);
        v[m] = make_float2(__uint_as_float(w.x ^ msk[m].x), __uint_as_float(w.y ^ msk[m].y));
      }
    }
  }
  // ---- phase A: butterfly over pair-index bits log2(L)..log2(L)+2 ----
  butterfly8<8>(v);
  // ---- transpose within the warp: lane l now owns pairs 8l..8l+7 ----
  uint8_t* tpb = smem + C::OFF_TP;
  if constexpr (L > 1) {
#pragma unroll
    for (int m = 0; m < 8; ++m) *reinterpret_cast<float2*>(tpb + G::tp(r, l + L * m)) = v[m];
    __syncwarp();
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 t = *reinterpret_cast<const float4*>(tpb + G::tp(r, 8 * l + 2 * q));
      v[2 * q] = make_float2(t.x, t.y);
      v[2 * q + 1] = make_float2(t.z, t.w);
    }
    // ---- phase B: butterfly over pair-index bits 0..log2(L)-1 (phase A did the rest) ----
    butterfly8<L>(v);
  }

  // ---- pass 1: pair energies s_j = E^2 + O^2 (r^2 = 2 s / d), row min/max ----
  float s[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) s[j] = __fmaf_rn(v[j].x, v[j].x, __fmul_rn(v[j].y, v[j].y));
  float smin = min3(min3(s[0], s[1], s[2]), min3(s[3], s[4], s[5]), fminf(s[6], s[7]));
  float smax = max3(max3(s[0], s[1], s[2]), max3(s[3], s[4], s[5]), fmaxf(s[6], s[7]));
#pragma unroll
  for (int off = 1; off < L; off <<= 1) {
    smin = fminf(smin, __shfl_xor_sync(0xffffffffu, smin, off));
    smax = fmaxf(smax, __shfl_xor_sync(0xffffffffu, smax, off));
  }
  const bool zero_row = !(smax > 0.f);

  // ---- row constants: stored header (Sec. 3.3), Eq. 2 scale, certification bound ----
  const float k2 = 2.0f / (float)D;
  float hmin, hmax, qscale, qbase, sfloor = 0.f;
  if (J.mode == TAC_NORM_LINEAR) {
    hmin = sqrt_approx(smin * k2);
    hmax = sqrt_approx(smax * k2);
    qscale = (float)Lq * rcp_approx(hmax - hmin);
    qbase = hmin;
  } else {  // log-space: norms floored at 2^-24 r_max
    sfloor = smax * 3.5527136788005009e-15f;  // 2^-48 on the energy
    hmin = sqrt_approx(fmaxf(smin, sfloor) * k2);
    hmax = sqrt_approx(smax * k2);
    const float lmin = lg2_approx(hmin);
    qscale = (float)Lq * rcp_approx(lg2_approx(hmax) - lmin);
    qbase = lmin;
  }
  if (!(hmax > hmin) || !(qscale <= 3.0e38f)) qscale = 0.f;
  // |dE|, |dO| <= (log2 d - 1) u ||x||_1 with ||x||_1 <= sqrt(d) ||x||_2 <= sqrt(d smax);
  // edge direction (1 ulp), product and fma add <= 4 u (|E| + |O|) <= 4 u sqrt(2 smax).
  const float rmx = sqrt_approx(smax);
  const float ty = (float)(G::LOGD - 1) * kU * 1.002f * sqrt_approx((float)D) * rmx;
  const float tau = ty + 5.f * kU * 1.4143f * rmx;
  // Pairs whose norm is so small that the fp32 angle may be off by a quarter bin
  // are re-decided too: sqrt(s) < 4 n ty / pi.
  const float rthr = ty * (4.f * (float)n / 3.14159265f);
  const float sthr = rthr * rthr;

  // ---- pass 2: angle codes (Alg. 1), norm codes (Eq. 2), packing ----
  const float2* et = reinterpret_cast<const float2*>(smem + C::OFF_TAB) + tab_offset(W);
  const float nb = (float)n * 0.15915494309189535f;  // bins per radian
  const float c1 = (0.78539816f + 0.273f) * nb;       // atan(t) ~ t (pi/4 + 0.273 (1 - t))
  const float c2 = 0.273f * nb;
  uint64_t acc_a = 0, acc_n = 0;
  uint32_t fm = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const float E = v[j].x, O = v[j].y;
    const float aE = fabsf(E), aO = fabsf(O);
    const float mx = fmaxf(aE, aO), mn = fminf(aE, aO);
    const float t = mn * rcp_approx(mx);
    const float phi = t * __fmaf_rn(t, -c2, c1);                 // octant angle, bins
    float fb = (aO > aE) ? (0.25f * n - phi) : phi;              // angle of (|E|, |O|)
    fb = (E < 0.f) ? (0.5f * n - fb) : fb;                       // angle of (E, |O|)
    const float ab = __uint_as_float(__float_as_uint(fb) ^ (__float_as_uint(O) & 0x80000000u));
    // theta = pi/4 - angle(E, O): candidate v - 1/2 rounded to an integer edge index
    const float vm = (0.125f * n - 0.5f) - ab;
    const int e = (__float_as_int(vm + 12582912.0f) - 0x4B400000) & (n - 1);
    const float2 dir = et[e];
    const float m = __fmaf_rn(E, dir.x, -__fmul_rn(O, dir.y));
    const int k = (e + 1 + (__float_as_int(m) >> 31)) & (n - 1);
    if (fabsf(m) < tau) fm |= 1u << j;
    float val;
    if (J.mode == TAC_NORM_LINEAR) val = sqrt_approx(s[j] * k2);
    else val = 0.5f * lg2_approx(fmaxf(s[j], sfloor) * k2);
    int c = __float2int_rd(__fmaf_rn(val - qbase, qscale, 0.5f));
    c = min(max(c, 0), Lq);
    acc_a |= (uint64_t)(uint32_t)k << (j * W);
    acc_n |= (uint64_t)(uint32_t)c << (j * B);
  }
  if (zero_row) { acc_a = 0; acc_n = 0; fm = 0; hmin = 0.f; hmax = 0.f; }
  else if (smin < sthr) {
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (s[j] < sthr) fm |= 1u << j;
  }
  if (!live) fm = 0;

  // ---- stage the records ----
  if (live) {
    store_bytes<W>(smem + C::OFF_ANG + r * AB + l * W, acc_a);
    store_bytes<B>(smem + C::OFF_NRM + r * NB + l * B, acc_n);
    if (l == 0) reinterpret_cast<float2*>(smem + C::OFF_HDR)[r] = make_float2(hmin, hmax);
  }
  __syncwarp();

  // ---- exact re-decision of the uncertified pairs, one warp per pair ----
  const int lane = tid & 31;
  const int wtid0 = tid & ~31;
  unsigned ball = __ballot_sync(0xffffffffu, fm != 0u);
  while (ball) {
    const int owner = __ffs(ball) - 1;
    ball &= ball - 1;
    uint32_t mm = __shfl_sync(0xffffffffu, fm, owner);
    const int otid = wtid0 + owner;
    const int rr = otid / L, ol = otid % L;
    while (mm) {
      const int j = __ffs(mm) - 1;
      mm &= mm - 1;
      const int i = 8 * ol + j;
      const int k = exact_angle_code<D, TIn>(J, in, rr, i, lane);
      if (lane == 0) patch_code(smem + C::OFF_ANG + rr * AB, i, W, k);
    }
    __syncwarp();
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
  } else {
    for (int rr = tid; rr < nrows; rr += kThreads) {
      const int64_t s = J.slot[row0 + rr];
      if (s < 0 || s >= J.capacity) continue;  // out-of-range slots are skipped
      copy_record<AB>(J.codes + s * AB, smem + C::OFF_ANG + rr * AB);
      copy_record<NB>(J.norms + s * NB, smem + C::OFF_NRM + rr * NB);
      reinterpret_cast<float2*>(J.hdr)[s] = reinterpret_cast<const float2*>(smem + C::OFF_HDR)[rr];
    }
  }
}

template <int D, typename TIn>
__global__ void __launch_bounds__(kThreads, 3) encode_kernel(const __grid_constant__ EncParams p) {
  using C = Enc<D, TIn>;
  using IT = typename C::IT;
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
  int mask_jid = -1;
  uint2 msk[8];
  // Prologue: kStages - 1 tiles in flight (one cp.async group per tile, possibly empty).
#pragma unroll
  for (int s = 0; s < kStages - 1; ++s) {
    const int ts = t + s * G;
    if (ts < p.ntiles) {
      const EncJob& Js = p.job[find_job(p, ts)];
      issue_tile_load<D, TIn>(Js, (ts - Js.tile0) * C::TR, smem + C::OFF_IN + s * IT::BYTES, tid);
    }
    cp_async_commit();
  }

  int cur = 0;
  for (; t < p.ntiles; t += G) {
    cp_async_wait<kStages - 2>();   // this tile's group has landed
    __syncthreads();                // ... and every thread is done with the previous tile
    {
      // Refill the buffer of the previous tile with the tile kStages - 1 ahead.
      const int tn = t + (kStages - 1) * G;
      int nb = cur + kStages - 1;
      if (nb >= kStages) nb -= kStages;
      if (tn < p.ntiles) {
        const EncJob& Jn = p.job[find_job(p, tn)];
        issue_tile_load<D, TIn>(Jn, (tn - Jn.tile0) * C::TR, smem + C::OFF_IN + nb * IT::BYTES, tid);
      }
      cp_async_commit();
    }
    const EncJob& J = p.job[jid];
    if (jid != mask_jid) {
      const int l = tid % C::L;
#pragma unroll
      for (int m = 0; m < 8; ++m) msk[m] = pair_sign_mask<C::ESZ>(J.signs, l + C::L * m);
      mask_jid = jid;
    }
    const int row0 = (t - J.tile0) * C::TR;
    const int nrows = (int)min((int64_t)C::TR, J.rows - row0);
    const uint8_t* in = smem + C::OFF_IN + cur * IT::BYTES;

#define TAC_ENC_CASE(WW)                                                          \
  case WW:                                                                        \
    if (J.b == 8) tile_body<D, TIn, WW, 8>(J, smem, in, nrows, tid, msk);         \
    else tile_body<D, TIn, WW, 4>(J, smem, in, nrows, tid, msk);                  \
    break;
    switch (J.w) {
      TAC_ENC_CASE(1) TAC_ENC_CASE(2) TAC_ENC_CASE(3) TAC_ENC_CASE(4)
      TAC_ENC_CASE(5) TAC_ENC_CASE(6) TAC_ENC_CASE(7) TAC_ENC_CASE(8)
      default: break;
    }
#undef TAC_ENC_CASE
    __syncthreads();

#define TAC_OUT_CASE(WW)                                                          \
  case WW:                                                                        \
    if (J.b == 8) copy_tile_out<D, TIn, WW, 8>(J, smem, row0, nrows, tid);        \
    else copy_tile_out<D, TIn, WW, 4>(J, smem, row0, nrows, tid);                 \
    break;
    switch (J.w) {
      TAC_OUT_CASE(1) TAC_OUT_CASE(2) TAC_OUT_CASE(3) TAC_OUT_CASE(4)
      TAC_OUT_CASE(5) TAC_OUT_CASE(6) TAC_OUT_CASE(7) TAC_OUT_CASE(8)
      default: break;
    }
#undef TAC_OUT_CASE

    if (t + G < p.ntiles) jid = find_job(p, t + G);
    cur = (cur + 1 == kStages) ? 0 : cur + 1;
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
