// TurboAngle decode kernel for sm_103a (Sec. 3.1 reconstruction with the Eq. 2
// dequantization of arXiv 2603.27467).
//
// One kernel per (d, output dtype, n = 2^W, norm bits B, norm mode), like the
// encoder.  A warp decodes warp tiles of RW = 32/L rows, L = d/16 lanes per
// row, 8 angle pairs per lane, each warp with its own pipeline:
//   1. a kNS-stage cp.async ring stages the tile's records (angle / norm /
//      header segments, each a whole number of 16-byte chunks): one chunk per
//      lane for contiguous slots, per-row copies for gathered slots;
//   2. lane l unpacks its 8 consecutive codes (pairs 8l..8l+7) and rebuilds each
//      pair from its bin-centre angle by table lookup: the table holds
//      (cos phi_k + sin phi_k, cos phi_k - sin phi_k) / sqrt(d), i.e. the
//      element-pair butterfly stage and the 1/sqrt(d) normalization are folded
//      into the lookup, so the remaining butterfly stages run straight from
//      (E_i, O_i) = r^_i * T[k_i] on packed fp32 pairs (FADD2/FFMA2): the low
//      pair-index bits in registers, an intra-warp shared-memory transpose, the
//      high bits;
//   3. D is a sign XOR on the output bits (after bf16 round-to-nearest-even, or
//      on fp32); each lane stores its pairs straight from registers: the L
//      lanes of a row write L consecutive pairs, whole 32-byte sectors.
#include <atomic>

#include "tac_common.cuh"

namespace tac {

constexpr int kNS = 4;  // pipeline stages per warp: kNS - 1 warp tiles of records in flight

__host__ __device__ constexpr int ilog2(int v) { return v <= 1 ? 0 : 1 + ilog2(v >> 1); }


// Shape of one kernel: n bins (W = ceil(log2 n) bits per code), B norm bits
// (4, 8, or 32 for fp32 norms), MODE; HB header bytes per row (none for fp32).
template <int D, typename TOut, int N, int B, int MODE>
struct Dec {
  using G = Geo<D>;
  static constexpr int P = G::P, L = G::L, RW = G::RW;
  static constexpr int ESZ = (int)sizeof(TOut);
  static constexpr int n = N;
  static constexpr int W = code_bits(N);
  static constexpr int AB = P * W / 8;        // angle record bytes per row
  static constexpr int NB = P * B / 8;        // norm record bytes per row
  static constexpr int HB = (MODE == TAC_NORM_FP32) ? 0 : 8;
  static constexpr int NA = RW * AB / 16, NN = RW * NB / 16, NH = RW * HB / 16;
  static constexpr int NCH = NA + NN + NH;
  static constexpr int ROUNDS = (NCH + 31) / 32;
  // one record stage of a warp tile: angle | norm | header segments
  static constexpr int R_ANG = 0;
  static constexpr int R_NRM = RW * AB;
  static constexpr int R_HDR = R_NRM + RW * NB;
  static constexpr int REC_W = R_HDR + RW * HB + 16;        // + slack for 3-word angle reads
  // per-warp shared memory region
  static constexpr int W_REC = 0;                           // kNS record stages
  static constexpr int W_TP = W_REC + kNS * REC_W;          // transpose rows
  static constexpr int WARP_B = W_TP + G::TP_W;
  static constexpr int TAB_E = 8;                           // one (float2) centre-table entry
  static constexpr int TABR = tab_copies(n, 16384);          // centre table copies
  // CTA shape: 8 warps, two CTAs per SM (up to 128 registers a thread; 10
  // warps at up to 102 registers measured 1.5 % slower).
  static constexpr int WARPS = 8;
  static constexpr int THREADS = 32 * WARPS;
  static constexpr int OFF_TAB = WARPS * WARP_B;            // centre table of this n (TABR copies)
  static constexpr int SMEM = OFF_TAB + n * TABR * TAB_E;
  static_assert(REC_W % 16 == 0 && W_TP % 16 == 0 && WARP_B % 16 == 0, "alignment");
};

// Stage the records of a tail tile (nrows < RW) or of gathered slots into
// `stage`.  Contiguous slots: 16-byte cp.async chunks of the three segments,
// the last chunk of each zero-filled past the tile.  Gathered slots: lane
// r < nrows copies row r's record with plain loads; an out-of-range slot
// decodes as an all-zero record.
template <int AB, int NB, int HB, int R_NRM, int R_HDR>
__device__ __noinline__ void stage_records_slow(const DecJob& J, int64_t row0, int nrows, uint8_t* stage,
                                                int lane) {
  if (J.slot == nullptr) {
    const int ba = nrows * AB, bn = nrows * NB, bh = nrows * HB;
    const int ca = (ba + 15) >> 4, cn = (bn + 15) >> 4, ch = (bh + 15) >> 4;
    const uint8_t* ga = J.codes + row0 * AB;
    const uint8_t* gn = J.norms + row0 * NB;
    const uint8_t* gh = J.hdr + row0 * 8;
    for (int q = lane; q < ca + cn + ch; q += 32) {
      if (q < ca) {
        const int rem = ba - 16 * q;
        cp_async16(stage + 16 * q, ga + 16 * q, rem >= 16 ? 16 : rem);
      } else if (q < ca + cn) {
        const int qq = q - ca, rem = bn - 16 * qq;
        cp_async16(stage + R_NRM + 16 * qq, gn + 16 * qq, rem >= 16 ? 16 : rem);
      } else {
        const int qq = q - ca - cn, rem = bh - 16 * qq;
        cp_async16(stage + R_HDR + 16 * qq, gh + 16 * qq, rem >= 16 ? 16 : rem);
      }
    }
  } else if (lane < nrows) {
    const int64_t s = J.slot[row0 + lane];
    uint8_t* da = stage + lane * AB;
    uint8_t* dn = stage + R_NRM + lane * NB;
    float2* dh = reinterpret_cast<float2*>(stage + R_HDR) + lane;
    if (s < 0 || s >= J.capacity) {
      for (int q = 0; q < AB; ++q) da[q] = 0;
      for (int q = 0; q < NB; ++q) dn[q] = 0;
      if constexpr (HB > 0) *dh = make_float2(0.f, 0.f);
      return;
    }
    const uint8_t* sa = J.codes + s * AB;
    const uint8_t* sn = J.norms + s * NB;
    if constexpr ((AB & 3) == 0) {
      for (int q = 0; q < AB / 4; ++q)
        reinterpret_cast<uint32_t*>(da)[q] = __ldg(reinterpret_cast<const uint32_t*>(sa) + q);
    } else {
      for (int q = 0; q < AB; ++q) da[q] = __ldg(sa + q);
    }
    for (int q = 0; q < NB / 4; ++q)
      reinterpret_cast<uint32_t*>(dn)[q] = __ldg(reinterpret_cast<const uint32_t*>(sn) + q);
    if constexpr (HB > 0) *dh = __ldg(reinterpret_cast<const float2*>(J.hdr) + s);
  }
}

// Read NBYTES (<= 8) bytes starting at shared byte address p (any alignment).
template <int NBYTES>
__device__ __forceinline__ uint64_t load_bytes(const uint8_t* p) {
  if constexpr (NBYTES == 8) {
    const uint2 t = *reinterpret_cast<const uint2*>(p);
    return (uint64_t)t.x | ((uint64_t)t.y << 32);
  } else if constexpr (NBYTES == 4) {
    return *reinterpret_cast<const uint32_t*>(p);
  } else {
    const uintptr_t a = reinterpret_cast<uintptr_t>(p);
    const uint32_t* w = reinterpret_cast<const uint32_t*>(a & ~(uintptr_t)3);
    const int sh = (int)(a & 3) * 8;
    const uint64_t lo = (uint64_t)w[0] | ((uint64_t)w[1] << 32);
    uint64_t v = lo >> sh;
    if (sh) v |= (uint64_t)w[2] << (64 - sh);
    return v;
  }
}

// Decode this lane's 8 pairs of warp-tile row r and store them (ttab: this
// lane's copy of the replicated centre table; orow: the lane's first output
// pair, element 2l of its row; live: the row exists).
template <int D, typename TOut, int N, int B, int MODE>
__device__ __forceinline__ void decode_body(const uint8_t* rec, uint8_t* wsm, const float2* ttab, int lane,
                                            const uint2 (&msk)[8], uint8_t* orow, bool live) {
  using C = Dec<D, TOut, N, B, MODE>;
  using G = Geo<D>;
  constexpr int L = C::L;
  constexpr int n = N, W = C::W;
  constexpr int AB = C::AB, NB = C::NB;
  const int r = lane / L, l = lane % L;

  const uint64_t acc_a = load_bytes<W>(rec + C::R_ANG + r * AB + l * W);
  // Code j's table entry: the W-bit field shifted straight to bit TSH (one
  // entry = TABR copies of TAB_E bytes), masked and OR'd with this lane's copy
  // offset: the byte offset of the entry in one shift and one logic op.  A
  // code of a non-power-of-two n is < n in every record this library writes;
  // clamping keeps any other record's table reads in bounds.
  constexpr int TSH = ilog2(C::TABR * C::TAB_E);
  const uint32_t lane_off = (uint32_t)((lane % C::TABR) * C::TAB_E);
  const uint8_t* tb = reinterpret_cast<const uint8_t*>(ttab);
  auto entry = [&](int j) -> float2 {
    const int pos = j * W;
    const uint32_t x = pos >= TSH ? (uint32_t)(acc_a >> (pos - TSH)) : (uint32_t)acc_a << (TSH - pos);
    uint32_t o = (x & ((uint32_t)((1 << W) - 1) << TSH)) | lane_off;
    if constexpr (!is_pow2(N)) o = min(o, ((uint32_t)(n - 1) << TSH) | lane_off);
    return *reinterpret_cast<const float2*>(tb + o);
  };
  float2 v[8];
  if constexpr (MODE == TAC_NORM_FP32) {  // r^ = the stored fp32 norm (Sec. 3.1)
    const float4* rp = reinterpret_cast<const float4*>(rec + C::R_NRM + r * NB + l * 32);
    const float4 a = rp[0], b = rp[1];
    const float rr[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = mul2(make_float2(rr[j], rr[j]), entry(j));
  } else {
  constexpr int Lq = (1 << B) - 1;
  const uint64_t acc_n = load_bytes<B>(rec + C::R_NRM + r * NB + l * B);
  const float2 h = reinterpret_cast<const float2*>(rec + C::R_HDR)[r];
  const float hmin = h.x, hmax = h.y;

  // Dequantization (the inverse of Eq. 2): linear r^ = r_min + c (r_max - r_min)/L,
  // log r^ = 2^(l_min + c (l_max - l_min)/L); r_max == r_min gives r^ = r_min.
  // The code enters as the float f = 1 + c 2^-B (its bits placed in the mantissa
  // of 1.0), so base + c step = fma(f, 2^B step, base - 2^B step).
  const bool spread = hmax > hmin;
  float base, step;
  if constexpr (MODE == TAC_NORM_LINEAR) {
    base = hmin;
    step = spread ? (hmax - hmin) * (1.0f / (float)Lq) : 0.f;
  } else {
    base = lg2_approx(hmin);
    step = spread ? (lg2_approx(hmax) - base) * (1.0f / (float)Lq) : 0.f;
  }
  const float S = step * (float)(1 << B);
  const float base2 = base - S;

#pragma unroll
  for (int j = 0; j < 8; ++j) {
    // norm code j shifted straight into the mantissa position 23 - B
    constexpr int NSH = 23 - B;
    const int pos = j * B;
    const uint32_t x = pos >= NSH ? (uint32_t)(acc_n >> (pos - NSH)) : (uint32_t)acc_n << (NSH - pos);
    const float f = __uint_as_float(0x3F800000u | (x & ((uint32_t)Lq << NSH)));
    float rh = __fmaf_rn(f, S, base2);
    if constexpr (MODE != TAC_NORM_LINEAR) rh = ex2_ftz(rh);
    v[j] = mul2(make_float2(rh, rh), entry(j));
  }
  }
  // Butterfly stages on pair-index bits 0..2 (this lane holds pairs 8l..8l+7).
  butterfly8<8>(v);
  if constexpr (L > 1) {
    uint8_t* tpr = wsm + C::W_TP + r * G::ST;
    uint8_t* tpl = tpr + (8 / L) * l * G::SM;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      *reinterpret_cast<float4*>(tpl + G::tp_pair((2 * q) ^ G::swb(l))) =
          make_float4(v[2 * q].x, v[2 * q].y, v[2 * q + 1].x, v[2 * q + 1].y);
    __syncwarp();
#pragma unroll
    for (int m = 0; m < 8; ++m) v[m] = *reinterpret_cast<const float2*>(tpr + m * G::SM + 8 * (l ^ G::swa(m)));
    // Stages on pair-index bits 3..log2(P)-1 (this lane now holds pairs l + L*m).
    butterfly8<8, 8 / L>(v);
  }
  // D, convert, store.  Record order: slot l + L*m is pair 4l + (m & 3) +
  // 4L (m >> 2), so a lane stores two runs of 4 pairs and the L lanes of a row
  // fill two whole lines (d = 128, bf16) per pair of store instructions.
  if constexpr (run_layout<D>()) {
    if (live) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        uint8_t* run = orow + h * 8 * C::ESZ * L;
        if constexpr (C::ESZ == 2) {
          uint32_t w[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const __nv_bfloat162 bb = __floats2bfloat162_rn(v[4 * h + j].x, v[4 * h + j].y);
            w[j] = (*reinterpret_cast<const uint32_t*>(&bb)) ^ msk[4 * h + j].x;
          }
          *reinterpret_cast<uint4*>(run) = make_uint4(w[0], w[1], w[2], w[3]);
        } else {
#pragma unroll
          for (int k = 0; k < 2; ++k) {
            const int m0 = 4 * h + 2 * k;
            *reinterpret_cast<uint4*>(run + 16 * k) =
                make_uint4(__float_as_uint(v[m0].x) ^ msk[m0].x, __float_as_uint(v[m0].y) ^ msk[m0].y,
                           __float_as_uint(v[m0 + 1].x) ^ msk[m0 + 1].x, __float_as_uint(v[m0 + 1].y) ^ msk[m0 + 1].y);
          }
        }
      }
    }
    return;
  }
  // Natural order (d <= 32): pair i = l + L*m; the L lanes of a row store L
  // consecutive pairs per instruction.
  if (live) {
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      if constexpr (C::ESZ == 2) {
        const __nv_bfloat162 bb = __floats2bfloat162_rn(v[m].x, v[m].y);
        *reinterpret_cast<uint32_t*>(orow + 4 * L * m) = (*reinterpret_cast<const uint32_t*>(&bb)) ^ msk[m].x;
      } else {
        *reinterpret_cast<uint2*>(orow + 8 * L * m) =
            make_uint2(__float_as_uint(v[m].x) ^ msk[m].x, __float_as_uint(v[m].y) ^ msk[m].y);
      }
    }
  }
}

template <int D, typename TOut, int N, int B, int MODE>
// Two CTAs per SM, as for the encoder: the scheduling room is worth more than
// a third CTA of warps.
__global__ void __launch_bounds__(Dec<D, TOut, N, B, MODE>::THREADS, kMinBlocks)
    decode_kernel(const __grid_constant__ DecParams p) {
  using C = Dec<D, TOut, N, B, MODE>;
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;

  // Centre table of this n: (cos + sin, cos - sin)(2 pi k / n) / sqrt(d).
  float2* ttab = reinterpret_cast<float2*>(smem + C::OFF_TAB);
  const float sc = sqrtf(2.f / (float)D);  // sqrt2 / sqrt(d)
  for (int k = tid; k < C::n; k += C::THREADS) {
    const float2 cs = cos_sin_q8(centre_q8(k, C::n), C::n);  // (cos psi, sin psi), psi = phi + pi/4
    const float2 e = make_float2(sc * cs.y, sc * cs.x);
#pragma unroll
    for (int c = 0; c < C::TABR; ++c) ttab[k * C::TABR + c] = e;
  }
  __syncthreads();

  // Each warp owns a contiguous range of warp tiles (balanced to +-1 tile).
  const int Gw = gridDim.x * C::WARPS, gw = blockIdx.x * C::WARPS + warp;
  const int per = p.ntiles / Gw, extra = p.ntiles % Gw;
  int t = gw * per + min(gw, extra);
  const int t_end = t + per + (gw < extra ? 1 : 0);
  if (t >= t_end) return;
  uint8_t* wsm = smem + warp * C::WARP_B;

  // ---- prefetch cursor: the next warp tile whose records are staged ----
  int it = t;                    // next tile to issue
  int pj = find_job(p, t);       // its job
  int p_end = 0;
  int64_t i_row0 = 0;            // the tile's first row within its job
  int64_t i_left = 0;            // rows of the job from i_row0
  bool p_dense = true;
  const uint8_t* i_src[C::ROUNDS];  // this lane's record chunk(s) of the tile
  int i_step[C::ROUNDS];            // bytes between consecutive tiles of its plane
  auto set_issue_job = [&]() {
    const DecJob& J = p.job[pj];
    p_end = (pj + 1 < p.njobs) ? p.job[pj + 1].tile0 : p.ntiles;
    const int rel = it - J.tile0;
    i_row0 = (int64_t)rel * C::RW;
    i_left = J.rows - i_row0;
    p_dense = J.slot == nullptr;
#pragma unroll
    for (int q = 0; q < C::ROUNDS; ++q) {
      const int ch = q * 32 + lane;
      if (ch < C::NA) { i_src[q] = J.codes + 16 * ch; i_step[q] = C::RW * C::AB; }
      else if (ch < C::NA + C::NN) { i_src[q] = J.norms + 16 * (ch - C::NA); i_step[q] = C::RW * C::NB; }
      else { i_src[q] = J.hdr + 16 * (ch - C::NA - C::NN); i_step[q] = C::RW * C::HB; }
      i_src[q] += (int64_t)rel * i_step[q];
    }
  };
  set_issue_job();
  auto issue = [&](int stg) {
    if (it < t_end) {
      if (it >= p_end) {  // a warp's tiles only move forward
        while (it >= p_end) { ++pj; p_end = (pj + 1 < p.njobs) ? p.job[pj + 1].tile0 : p.ntiles; }
        set_issue_job();
      }
      uint8_t* stage = wsm + C::W_REC + stg * C::REC_W;
      if (p_dense && i_left >= C::RW) {
#pragma unroll
        for (int q = 0; q < C::ROUNDS; ++q) {
          const int ch = q * 32 + lane;
          if (ch < C::NCH) cp_async16(stage + 16 * ch, i_src[q], 16);
        }
      } else {
        stage_records_slow<C::AB, C::NB, C::HB, C::R_NRM, C::R_HDR>(p.job[pj], i_row0, (int)min((int64_t)C::RW, i_left),
                                                            stage, lane);
      }
#pragma unroll
      for (int q = 0; q < C::ROUNDS; ++q) i_src[q] += i_step[q];
      i_row0 += C::RW;
      i_left -= C::RW;
      ++it;
    }
    cp_async_commit();
  };
#pragma unroll
  for (int s = 0; s < kNS - 1; ++s) issue(s);

  // ---- compute cursor ----
  int c_end = t;                 // first tile after the current job (forces a job load)
  int64_t c_left = 0;            // rows of the job from the current tile's row 0
  int64_t c_step = 0;            // output bytes between consecutive tiles (RW rows)
  const int r = lane / C::L, l = lane % C::L;
  uint8_t* o_row = nullptr;      // this lane's first output pair in the current tile
  uint2 msk[8];
#pragma unroll
  for (int m = 0; m < 8; ++m) msk[m] = make_uint2(0u, 0u);

  static_assert((kNS & (kNS - 1)) == 0, "stage ring size");
  int stage = 0;
  // Iterations ahead that need no checks: the decoded tile is a full tile of
  // the current job and the prefetched tile a full tile of the (contiguous)
  // issue job inside the warp's range.  Set by the general iterations.
  int fast = 0;
  while (t < t_end) {
    if (fast > 0) {
      // A stretch of `fast` tiles, each a full tile of the current job whose
      // prefetch is a full tile of the (contiguous) issue job: no per-tile
      // checks, the cursors are settled once after it.
      const int t_stop = t + fast;
      for (; t < t_stop; ++t) {
        cp_async_wait<kNS - 2>();   // this warp tile's records have landed
        __syncwarp();               // ... and every lane is done with the previous tile
        uint8_t* dst = wsm + C::W_REC + ((stage + kNS - 1) & (kNS - 1)) * C::REC_W;
#pragma unroll
        for (int q = 0; q < C::ROUNDS; ++q) {
          const int ch = q * 32 + lane;
          if (ch < C::NCH) cp_async16(dst + 16 * ch, i_src[q], 16);
          i_src[q] += i_step[q];
        }
        cp_async_commit();
        decode_body<D, TOut, N, B, MODE>(wsm + C::W_REC + stage * C::REC_W, wsm, ttab, lane, msk, o_row, true);
        o_row += c_step;
        stage = (stage + 1) & (kNS - 1);
      }
      const int64_t adv = (int64_t)fast * C::RW;
      i_row0 += adv;
      i_left -= adv;
      it += fast;
      c_left -= adv;
      fast = 0;
      continue;
    }

    // ---- general tile: a job's first tile, tails, gathered slots, range ends ----
    cp_async_wait<kNS - 2>();
    __syncwarp();
    issue((stage + kNS - 1) & (kNS - 1));
    if (t >= c_end) {  // next job
      const int cj = find_job(p, t);
      const DecJob& J = p.job[cj];
      c_end = (cj + 1 < p.njobs) ? p.job[cj + 1].tile0 : p.ntiles;
      const int64_t row0 = (int64_t)(t - J.tile0) * C::RW;
      c_left = J.rows - row0;
      const int64_t sb = J.stride * C::ESZ;
      c_step = C::RW * sb;
      o_row = reinterpret_cast<uint8_t*>(J.y) + (row0 + r) * sb + (run_layout<D>() ? 8 : 2) * C::ESZ * l;
#pragma unroll
      for (int m = 0; m < 8; ++m) msk[m] = pair_sign_mask<C::ESZ>(J.signs, slot_pair<D>(l + C::L * m));
    }
    decode_body<D, TOut, N, B, MODE>(wsm + C::W_REC + stage * C::REC_W, wsm, ttab, lane, msk, o_row, r < c_left);
    o_row += c_step;
    c_left -= C::RW;
    stage = (stage + 1) & (kNS - 1);
    ++t;
    // c_left now counts the rows of the compute job from tile t, i_left those
    // of the issue job from tile it (the next to prefetch).
    const int64_t cf = c_left / C::RW;
    const int64_t pf = p_dense ? min(min((int64_t)(p_end - it), i_left / C::RW), (int64_t)(t_end - it)) : 0;
    const int64_t f = min(cf, pf);
    fast = f > 0 ? (int)f : 0;
  }
  cp_async_wait<0>();
}

template <int D, typename TOut, int N, int B, int MODE>
static cudaError_t launch_decode_v(const DecParams& p, int grid_cap, cudaStream_t st) {
  using C = Dec<D, TOut, N, B, MODE>;
  auto kern = decode_kernel<D, TOut, N, B, MODE>;
  static std::atomic<int> configured[64];   // per device; concurrent first calls set the same
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && configured[dev].load(std::memory_order_acquire) == 0) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    configured[dev].store(1, std::memory_order_release);
  }
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, C::THREADS, C::SMEM);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) per_sm = 1;
  int grid = grid_cap * per_sm;
  const int need = (p.ntiles + C::WARPS - 1) / C::WARPS;
  if (grid > need) grid = need;
  if (grid < 1) return cudaSuccess;
  kern<<<grid, C::THREADS, C::SMEM, st>>>(p);
  return cudaGetLastError();
}

// One kernel per supported (n, norm bits, mode), as for the encoder.
template <int D, typename TOut>
static cudaError_t launch_decode_t(const DecParams& p, int n, int b, int mode, int sms, cudaStream_t st) {
#define TAC_DEC_N(NN)                                                                                   \
  if (n == NN) {                                                                                        \
    if (mode == TAC_NORM_FP32) return b == 32 ? launch_decode_v<D, TOut, NN, 32, TAC_NORM_FP32>(p, sms, st) \
                                              : cudaErrorInvalidValue;                                  \
    if (b == 4) return mode == TAC_NORM_LOG ? launch_decode_v<D, TOut, NN, 4, TAC_NORM_LOG>(p, sms, st)    \
                                            : launch_decode_v<D, TOut, NN, 4, TAC_NORM_LINEAR>(p, sms, st); \
    if (b == 8) return mode == TAC_NORM_LOG ? launch_decode_v<D, TOut, NN, 8, TAC_NORM_LOG>(p, sms, st)    \
                                            : launch_decode_v<D, TOut, NN, 8, TAC_NORM_LINEAR>(p, sms, st); \
    return cudaErrorInvalidValue;                                                                       \
  }
  TAC_DEC_N(2) TAC_DEC_N(4) TAC_DEC_N(8) TAC_DEC_N(16) TAC_DEC_N(32) TAC_DEC_N(64) TAC_DEC_N(128)
  TAC_DEC_N(256) TAC_DEC_N(48) TAC_DEC_N(56)
#undef TAC_DEC_N
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
#define TAC_DEC_INSTANCE(DD, NAME, T)                                                                 \
  cudaError_t launch_decode_##DD##_##NAME(const DecParams& p, int n, int b, int mode, int sms,       \
                                          cudaStream_t st) {                                         \
    return launch_decode_t<DD, T>(p, n, b, mode, sms, st);                                           \
  }
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 16 && TAC_INST_BF16)
TAC_DEC_INSTANCE(16, bf16, __nv_bfloat16)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 32 && TAC_INST_BF16)
TAC_DEC_INSTANCE(32, bf16, __nv_bfloat16)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 64 && TAC_INST_BF16)
TAC_DEC_INSTANCE(64, bf16, __nv_bfloat16)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 128 && TAC_INST_BF16)
TAC_DEC_INSTANCE(128, bf16, __nv_bfloat16)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 16 && TAC_INST_F32)
TAC_DEC_INSTANCE(16, f32, float)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 32 && TAC_INST_F32)
TAC_DEC_INSTANCE(32, f32, float)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 64 && TAC_INST_F32)
TAC_DEC_INSTANCE(64, f32, float)
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 128 && TAC_INST_F32)
TAC_DEC_INSTANCE(128, f32, float)
#endif
#undef TAC_DEC_INSTANCE

}  // namespace tac
