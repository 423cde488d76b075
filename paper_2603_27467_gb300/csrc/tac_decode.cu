// TurboAngle decode kernel for sm_103a (Sec. 3.1 reconstruction with the Eq. 2
// dequantization of arXiv 2603.27467).
//
// A 256-thread CTA decodes a tile of TR = 256/L rows, L = d/16 lanes per row,
// 8 angle pairs per lane:
//   1. the tile's records (angle / norm / header planes) are staged global ->
//      shared with cp.async: coalesced 16-byte chunks for contiguous slots,
//      per-row copies for gathered slots; double buffered;
//   2. lane l unpacks its 8 consecutive codes (pairs 8l..8l+7) and rebuilds each
//      pair from its bin-centre angle by table lookup: the table holds
//      (cos phi_k + sin phi_k, cos phi_k - sin phi_k) / sqrt(d), i.e. the
//      element-pair butterfly stage and the 1/sqrt(d) normalization are folded
//      into the lookup, so the remaining butterfly stages run straight from
//      (E_i, O_i) = r^_i * T[k_i] on packed fp32 pairs (FADD2/FFMA2): the low
//      pair-index bits in registers, an intra-warp shared-memory transpose, the
//      high bits;
//   3. D is a sign XOR on the output bits (after bf16 round-to-nearest-even, or
//      on fp32); rows are staged in shared memory and written with coalesced
//      16-byte stores.
#include "tac_common.cuh"

namespace tac {

constexpr int kNS = 4;  // pipeline stages per warp: kNS - 1 warp tiles of records in flight

template <int D, typename TOut>
struct Dec {
  using G = Geo<D>;
  using OT = RowTile<D, (int)sizeof(TOut)>;
  static constexpr int P = G::P, L = G::L, RW = G::RW;
  static constexpr int ESZ = (int)sizeof(TOut);
  // one record stage of a warp tile: angle, norm and header segments
  static constexpr int R_ANG = 0;
  static constexpr int R_NRM = RW * P;                      // angle records <= P bytes per row
  static constexpr int R_HDR = R_NRM + RW * P;              // norm records <= P bytes per row
  static constexpr int REC_W = R_HDR + RW * 8 + 16;         // + slack for 3-word angle reads
  // per-warp shared memory region
  static constexpr int W_REC = 0;                           // kNS record stages
  static constexpr int W_TP = W_REC + kNS * REC_W;          // transpose rows
  static constexpr int W_OUT = W_TP + G::TP_W;              // output rows
  static constexpr int W_JOB = W_OUT + OT::BYTES;           // current job (DecWarpJob)
  static constexpr int WARP_B = W_JOB + 128;
  static constexpr int OFF_TAB = kWarps * WARP_B;           // centre tables, every n
  static constexpr int SMEM = OFF_TAB + kTabEntries * 8;
  static_assert(REC_W % 16 == 0 && W_OUT % 16 == 0 && W_JOB % 16 == 0, "alignment");
};

struct DecWarpJob {
  void* y;
  int64_t rows;
  int64_t stride;  // elements
  int32_t t0, end, variant, pad_;
};
static_assert(sizeof(DecWarpJob) <= 128, "DecWarpJob");

// Stage the records of warp tile (row0, nrows) of a job into `stage`.
// Contiguous slots: 16-byte cp.async chunks of the three plane segments (a
// segment of a full tile is a multiple of 16 bytes; a tail tile's last chunk is
// zero-filled).  Gathered slots: lane r < nrows copies row r's record with plain loads.
template <int D, typename TOut>
__device__ __forceinline__ void stage_records(const uint8_t* codes, const uint8_t* norms, const uint8_t* hdr,
                                              const int64_t* slot, int64_t capacity, int64_t row0, int nrows,
                                              int AB, int NB, uint8_t* stage, int lane) {
  using C = Dec<D, TOut>;
  if (slot == nullptr) {
    const int ba = nrows * AB, bn = nrows * NB, bh = nrows * 8;
    const int ca = (ba + 15) >> 4, cn = (bn + 15) >> 4, ch = (bh + 15) >> 4;
    const uint8_t* ga = codes + row0 * AB;
    const uint8_t* gn = norms + row0 * NB;
    const uint8_t* gh = hdr + row0 * 8;
    for (int q = lane; q < ca + cn + ch; q += 32) {
      if (q < ca) {
        const int rem = ba - 16 * q;
        cp_async16(stage + C::R_ANG + 16 * q, ga + 16 * q, rem >= 16 ? 16 : rem);
      } else if (q < ca + cn) {
        const int qq = q - ca, rem = bn - 16 * qq;
        cp_async16(stage + C::R_NRM + 16 * qq, gn + 16 * qq, rem >= 16 ? 16 : rem);
      } else {
        const int qq = q - ca - cn, rem = bh - 16 * qq;
        cp_async16(stage + C::R_HDR + 16 * qq, gh + 16 * qq, rem >= 16 ? 16 : rem);
      }
    }
  } else if (lane < nrows) {
    const int64_t s = slot[row0 + lane];
    uint8_t* da = stage + C::R_ANG + lane * AB;
    uint8_t* dn = stage + C::R_NRM + lane * NB;
    float2* dh = reinterpret_cast<float2*>(stage + C::R_HDR) + lane;
    if (s < 0 || s >= capacity) {  // out-of-range slot: decodes as an all-zero record
      for (int q = 0; q < AB; ++q) da[q] = 0;
      for (int q = 0; q < NB; ++q) dn[q] = 0;
      *dh = make_float2(0.f, 0.f);
      return;
    }
    const uint8_t* sa = codes + s * AB;
    const uint8_t* sn = norms + s * NB;
    if ((AB & 3) == 0) {
      for (int q = 0; q < AB / 4; ++q) reinterpret_cast<uint32_t*>(da)[q] = __ldg(reinterpret_cast<const uint32_t*>(sa) + q);
    } else {
      for (int q = 0; q < AB; ++q) da[q] = __ldg(sa + q);
    }
    for (int q = 0; q < NB / 4; ++q) reinterpret_cast<uint32_t*>(dn)[q] = __ldg(reinterpret_cast<const uint32_t*>(sn) + q);
    *dh = __ldg(reinterpret_cast<const float2*>(hdr) + s);
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

// Decode this lane's 8 pairs of warp-tile row r and stage the output row segment.
template <int D, typename TOut, int W, int B, int MODE>
__device__ __forceinline__ void decode_body(const uint8_t* rec, uint8_t* wsm, const float2* ttab_all, int lane,
                                            const uint2 (&msk)[8]) {
  using C = Dec<D, TOut>;
  using G = Geo<D>;
  using OT = typename C::OT;
  constexpr int P = C::P, L = C::L;
  constexpr int n = 1 << W;
  constexpr int AB = P * W / 8;
  constexpr int NB = P * B / 8;
  constexpr int Lq = (1 << B) - 1;
  const int r = lane / L, l = lane % L;
  const float2* ttab = ttab_all + tab_offset(W);

  const uint64_t acc_a = load_bytes<W>(rec + C::R_ANG + r * AB + l * W);
  const uint64_t acc_n = load_bytes<B>(rec + C::R_NRM + r * NB + l * B);
  const float2 h = reinterpret_cast<const float2*>(rec + C::R_HDR)[r];
  const float hmin = h.x, hmax = h.y;

  // Dequantization (the inverse of Eq. 2): linear r^ = r_min + c (r_max - r_min)/L,
  // log r^ = 2^(l_min + c (l_max - l_min)/L); r_max == r_min gives r^ = r_min.
  const bool spread = hmax > hmin;
  float base, step;
  if constexpr (MODE == TAC_NORM_LINEAR) {
    base = hmin;
    step = spread ? (hmax - hmin) * (1.0f / (float)Lq) : 0.f;
  } else {
    base = lg2_approx(hmin);
    step = spread ? (lg2_approx(hmax) - base) * (1.0f / (float)Lq) : 0.f;
  }

  float2 v[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const uint32_t k = (uint32_t)(acc_a >> (j * W)) & (uint32_t)(n - 1);
    const uint32_t c = (uint32_t)(acc_n >> (j * B)) & (uint32_t)Lq;
    float rh = __fmaf_rn(__uint2float_rn(c), step, base);
    if constexpr (MODE != TAC_NORM_LINEAR) rh = ex2_approx(rh);
    const float2 t = ttab[k];
    v[j] = make_float2(rh * t.x, rh * t.y);
  }
  // Butterfly stages on pair-index bits 0..2 (this lane holds pairs 8l..8l+7).
  butterfly8<8>(v);
  if constexpr (L > 1) {
    uint8_t* tpr = wsm + C::W_TP + r * G::ST;
    uint8_t* tpl = tpr + (8 / L) * l * G::SM;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      *reinterpret_cast<float4*>(tpl + G::tp_pair(2 * q)) =
          make_float4(v[2 * q].x, v[2 * q].y, v[2 * q + 1].x, v[2 * q + 1].y);
    __syncwarp();
#pragma unroll
    for (int m = 0; m < 8; ++m) v[m] = *reinterpret_cast<const float2*>(tpr + m * G::SM + 8 * l);
    // Stages on pair-index bits 3..log2(P)-1 (this lane now holds pairs l + L*m).
    butterfly8<8, 8 / L>(v);
  }
  // D, convert, stage the row: pair i = l + L*m is element pair (2i, 2i+1).
  uint8_t* orow = wsm + C::W_OUT + r * OT::STRIDE + 2 * C::ESZ * l;
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

template <int D, typename TOut>
__global__ void __launch_bounds__(kThreads, 3) decode_kernel(const __grid_constant__ DecParams p) {
  using C = Dec<D, TOut>;
  using OT = typename C::OT;
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;

  // Centre tables for every n = 2..256: (cos + sin, cos - sin)(2 pi k / n) / sqrt(d).
  float2* ttab = reinterpret_cast<float2*>(smem + C::OFF_TAB);
  const float sc = sqrtf(2.f / (float)D);  // sqrt2 / sqrt(d)
  for (int idx = tid; idx < kTabEntries - 2; idx += kThreads) {
    const int w = 31 - __clz(idx + 2);
    const int k = idx - tab_offset(w);
    const float2 cs = cos_sin_q8(centre_q8(k, 1 << w), 1 << w);  // (cos psi, sin psi), psi = phi + pi/4
    ttab[idx] = make_float2(sc * cs.y, sc * cs.x);
  }
  __syncthreads();

  const int Gw = gridDim.x * kWarps;
  int t = blockIdx.x * kWarps + warp;
  if (t >= p.ntiles) return;
  uint8_t* wsm = smem + warp * C::WARP_B;

  // Prefetch cursor: the job of the next warp tile whose records are staged.
  int pj = find_job(p, t);
  int p_end = (pj + 1 < p.njobs) ? p.job[pj + 1].tile0 : p.ntiles;
  auto issue = [&](int tt, int stg) {
    if (tt < p.ntiles) {
      while (tt >= p_end) {
        ++pj;
        p_end = (pj + 1 < p.njobs) ? p.job[pj + 1].tile0 : p.ntiles;
      }
      const DecJob& J = p.job[pj];
      const int64_t row0 = (int64_t)(tt - J.tile0) * C::RW;
      const int nrows = (int)min((int64_t)C::RW, J.rows - row0);
      stage_records<D, TOut>(J.codes, J.norms, J.hdr, J.slot, J.capacity, row0, nrows, C::P * J.w / 8,
                             C::P * J.b / 8, wsm + C::W_REC + stg * C::REC_W, lane);
    }
    cp_async_commit();
  };
#pragma unroll
  for (int s = 0; s < kNS - 1; ++s) issue(t + s * Gw, s);

  DecWarpJob* wj = reinterpret_cast<DecWarpJob*>(wsm + C::W_JOB);
  int cj = -1, c_end = 0;
  uint2 msk[8];
#pragma unroll
  for (int m = 0; m < 8; ++m) msk[m] = make_uint2(0u, 0u);

  int stage = 0;
  for (; t < p.ntiles; t += Gw) {
    cp_async_wait<kNS - 2>();   // this warp tile's records have landed
    __syncwarp();               // ... and every lane is done with the previous tile
    {
      int ns = stage + kNS - 1;
      if (ns >= kNS) ns -= kNS;
      issue(t + (kNS - 1) * Gw, ns);
    }
    if (t >= c_end) {  // next job: copy its descriptor to shared memory
      cj = (cj < 0) ? find_job(p, t) : cj + 1;
      while (cj + 1 < p.njobs && p.job[cj + 1].tile0 <= t) ++cj;
      const DecJob& J = p.job[cj];
      c_end = (cj + 1 < p.njobs) ? p.job[cj + 1].tile0 : p.ntiles;
      if (lane == 0) {
        wj->y = J.y; wj->rows = J.rows; wj->stride = J.stride; wj->t0 = J.tile0; wj->end = c_end;
        wj->variant = (J.w - 1) * 4 + (J.b == 8 ? 2 : 0) + (J.mode == TAC_NORM_LOG ? 1 : 0);
      }
      const int l = lane % C::L;
#pragma unroll
      for (int m = 0; m < 8; ++m) msk[m] = pair_sign_mask<C::ESZ>(J.signs, l + C::L * m);
      __syncwarp();
    }
    const uint8_t* rec = wsm + C::W_REC + stage * C::REC_W;

#define TAC_DEC_CASE(WW)                                                                              \
  case (WW - 1) * 4 + 0: decode_body<D, TOut, WW, 4, TAC_NORM_LINEAR>(rec, wsm, ttab, lane, msk); break;  \
  case (WW - 1) * 4 + 1: decode_body<D, TOut, WW, 4, TAC_NORM_LOG>(rec, wsm, ttab, lane, msk); break;     \
  case (WW - 1) * 4 + 2: decode_body<D, TOut, WW, 8, TAC_NORM_LINEAR>(rec, wsm, ttab, lane, msk); break;  \
  case (WW - 1) * 4 + 3: decode_body<D, TOut, WW, 8, TAC_NORM_LOG>(rec, wsm, ttab, lane, msk); break;
    switch (wj->variant) {
      TAC_DEC_CASE(1) TAC_DEC_CASE(2) TAC_DEC_CASE(3) TAC_DEC_CASE(4)
      TAC_DEC_CASE(5) TAC_DEC_CASE(6) TAC_DEC_CASE(7) TAC_DEC_CASE(8)
      default: break;
    }
#undef TAC_DEC_CASE
    __syncwarp();
    // Write the warp tile's rows: 16-byte chunks, coalesced.
    {
      const int64_t row0 = (int64_t)(t - wj->t0) * C::RW;
      const int nrows = (int)min((int64_t)C::RW, wj->rows - row0);
      uint8_t* y = reinterpret_cast<uint8_t*>(wj->y);
      const int64_t sb = wj->stride * C::ESZ;
#pragma unroll
      for (int q = 0; q < OT::CHUNKS; ++q) {
        const int id = q * 32 + lane;
        const int rr = id / OT::CPR, col = (id % OT::CPR) * 16;
        if (rr < nrows)
          *reinterpret_cast<uint4*>(y + (row0 + rr) * sb + col) =
              *reinterpret_cast<const uint4*>(wsm + C::W_OUT + rr * OT::STRIDE + col);
      }
    }
    stage = (stage + 1 == kNS) ? 0 : stage + 1;
  }
  cp_async_wait<0>();
}

template <int D, typename TOut>
static cudaError_t launch_decode_t(const DecParams& p, int grid_cap, cudaStream_t st) {
  using C = Dec<D, TOut>;
  auto kern = decode_kernel<D, TOut>;
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
  const int need = (p.ntiles + kWarps - 1) / kWarps;
  if (grid > need) grid = need;
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
cudaError_t launch_decode_16_bf16(const DecParams& p, int sms, cudaStream_t st) {
  return launch_decode_t<16, __nv_bfloat16>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 32 && TAC_INST_BF16)
cudaError_t launch_decode_32_bf16(const DecParams& p, int sms, cudaStream_t st) {
  return launch_decode_t<32, __nv_bfloat16>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 64 && TAC_INST_BF16)
cudaError_t launch_decode_64_bf16(const DecParams& p, int sms, cudaStream_t st) {
  return launch_decode_t<64, __nv_bfloat16>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 128 && TAC_INST_BF16)
cudaError_t launch_decode_128_bf16(const DecParams& p, int sms, cudaStream_t st) {
  return launch_decode_t<128, __nv_bfloat16>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 16 && TAC_INST_F32)
cudaError_t launch_decode_16_f32(const DecParams& p, int sms, cudaStream_t st) {
  return launch_decode_t<16, float>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 32 && TAC_INST_F32)
cudaError_t launch_decode_32_f32(const DecParams& p, int sms, cudaStream_t st) {
  return launch_decode_t<32, float>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 64 && TAC_INST_F32)
cudaError_t launch_decode_64_f32(const DecParams& p, int sms, cudaStream_t st) {
  return launch_decode_t<64, float>(p, sms, st);
}
#endif
#if defined(TAC_ALL_INSTANCES) || (TAC_INST_D == 128 && TAC_INST_F32)
cudaError_t launch_decode_128_f32(const DecParams& p, int sms, cudaStream_t st) {
  return launch_decode_t<128, float>(p, sms, st);
}
#endif

}  // namespace tac
