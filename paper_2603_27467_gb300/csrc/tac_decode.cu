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

constexpr int kStages = 4;  // record tiles per CTA: 3 in flight while one is decoded

template <int D, typename TOut>
struct Dec {
  using G = Geo<D>;
  using OT = RowTile<D, (int)sizeof(TOut)>;
  static constexpr int P = G::P, L = G::L, TR = G::TR;
  static constexpr int ESZ = (int)sizeof(TOut);
  static constexpr int ABMAX = P;                        // angle record bytes at w = 8
  static constexpr int NBMAX = P;                        // norm record bytes at b = 8
  static constexpr int R_ANG = 0;                        // inside a record buffer
  static constexpr int R_NRM = TR * ABMAX;
  static constexpr int R_HDR = R_NRM + TR * NBMAX;
  static constexpr int REC_B = R_HDR + TR * 8 + 16;      // + slack for 3-word angle reads
  // shared memory layout (bytes)
  static constexpr int OFF_REC = 0;                      // kStages record buffers
  static constexpr int OFF_TP = OFF_REC + kStages * REC_B; // transpose buffer
  static constexpr int OFF_OUT = OFF_TP + G::TP_B;       // output tile
  static constexpr int OFF_TAB = OFF_OUT + OT::BYTES;    // centre tables, every n
  static constexpr int SMEM = OFF_TAB + kTabEntries * 8;
  static constexpr int CHUNKS = TR * OT::CPR / kThreads;
  static_assert(TR * OT::CPR % kThreads == 0, "tile chunks");
  static_assert(REC_B % 16 == 0, "record buffer alignment");
};

// Cooperative cp.async of `bytes` contiguous bytes (16-byte aligned global base),
// zero-filling the tail of the last chunk.
__device__ __forceinline__ void cta_copy_in(uint8_t* s, const uint8_t* g, int bytes, int tid) {
  const int nch = (bytes + 15) >> 4;
  for (int q = tid; q < nch; q += kThreads) {
    const int rem = bytes - (q << 4);
    cp_async16(s + (q << 4), g + (q << 4), rem >= 16 ? 16 : rem);
  }
}

template <int D, typename TOut>
__device__ __forceinline__ void issue_rec_load(const DecJob& J, int row0, int nrows, uint8_t* buf, int tid) {
  using C = Dec<D, TOut>;
  const int AB = C::P * J.w / 8, NB = C::P * J.b / 8;
  if (J.slot == nullptr) {
    cta_copy_in(buf + C::R_ANG, J.codes + (int64_t)row0 * AB, nrows * AB, tid);
    cta_copy_in(buf + C::R_NRM, J.norms + (int64_t)row0 * NB, nrows * NB, tid);
    cta_copy_in(buf + C::R_HDR, J.hdr + (int64_t)row0 * 8, nrows * 8, tid);
  } else {
    // Gather: one thread per row copies its record byte-exactly with plain loads
    // (records of odd size are not 16-byte aligned in the source planes).
    for (int rr = tid; rr < nrows; rr += kThreads) {
      const int64_t s = J.slot[row0 + rr];
      uint8_t* da = buf + C::R_ANG + rr * AB;
      uint8_t* dn = buf + C::R_NRM + rr * NB;
      float2* dh = reinterpret_cast<float2*>(buf + C::R_HDR) + rr;
      if (s < 0 || s >= J.capacity) {  // out-of-range slot: decodes as an all-zero record
        for (int q = 0; q < AB; ++q) da[q] = 0;
        for (int q = 0; q < NB; ++q) dn[q] = 0;
        *dh = make_float2(0.f, 0.f);
        continue;
      }
      const uint8_t* sa = J.codes + s * AB;
      const uint8_t* sn = J.norms + s * NB;
      if ((AB & 3) == 0) {
        for (int q = 0; q < AB / 4; ++q) reinterpret_cast<uint32_t*>(da)[q] = __ldg(reinterpret_cast<const uint32_t*>(sa) + q);
      } else {
        for (int q = 0; q < AB; ++q) da[q] = __ldg(sa + q);
      }
      if ((NB & 3) == 0) {
        for (int q = 0; q < NB / 4; ++q) reinterpret_cast<uint32_t*>(dn)[q] = __ldg(reinterpret_cast<const uint32_t*>(sn) + q);
      } else {
        for (int q = 0; q < NB; ++q) dn[q] = __ldg(sn + q);
      }
      *dh = __ldg(reinterpret_cast<const float2*>(J.hdr) + s);
    }
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

template <int D, typename TOut, int W, int B>
__device__ __forceinline__ void decode_row(const DecJob& J, const uint8_t* rec, uint8_t* smem, int tid,
                                           const uint2 (&msk)[8]) {
  using C = Dec<D, TOut>;
  using G = Geo<D>;
  using OT = typename C::OT;
  constexpr int P = C::P, L = C::L;
  constexpr int n = 1 << W;
  constexpr int AB = P * W / 8;
  constexpr int NB = P * B / 8;
  constexpr int Lq = (1 << B) - 1;
  const int r = tid / L, l = tid % L;
  const float2* ttab = reinterpret_cast<const float2*>(smem + C::OFF_TAB) + tab_offset(W);

  const uint64_t acc_a = load_bytes<W>(rec + C::R_ANG + r * AB + l * W);
  const uint64_t acc_n = load_bytes<B>(rec + C::R_NRM + r * NB + l * B);
  const float2 h = reinterpret_cast<const float2*>(rec + C::R_HDR)[r];
  const float hmin = h.x, hmax = h.y;

  // Dequantization (the inverse of Eq. 2): linear r^ = r_min + c (r_max - r_min)/L,
  // log r^ = 2^(l_min + c (l_max - l_min)/L); r_max == r_min gives r^ = r_min.
  const bool spread = hmax > hmin;
  float base, step;
  if (J.mode == TAC_NORM_LINEAR) {
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
    if (J.mode != TAC_NORM_LINEAR) rh = ex2_approx(rh);
    const float2 t = ttab[k];
    v[j] = make_float2(rh * t.x, rh * t.y);
  }
  // Butterfly stages on pair-index bits 0..2 (this lane holds pairs 8l..8l+7).
  butterfly8<8>(v);
  if constexpr (L > 1) {
    uint8_t* tpb = smem + C::OFF_TP;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      *reinterpret_cast<float4*>(tpb + G::tp(r, 8 * l + 2 * q)) =
          make_float4(v[2 * q].x, v[2 * q].y, v[2 * q + 1].x, v[2 * q + 1].y);
    __syncwarp();
#pragma unroll
    for (int m = 0; m < 8; ++m) v[m] = *reinterpret_cast<const float2*>(tpb + G::tp(r, l + L * m));
    // Stages on pair-index bits 3..log2(P)-1 (this lane now holds pairs l + L*m).
    butterfly8<8, 8 / L>(v);
  }
  // D, convert, stage the row: pair i = l + L*m is element pair (2i, 2i+1).
  uint8_t* orow = smem + C::OFF_OUT + r * OT::STRIDE;
#pragma unroll
  for (int m = 0; m < 8; ++m) {
    const int i = l + L * m;
    if constexpr (C::ESZ == 2) {
      const __nv_bfloat162 bb = __floats2bfloat162_rn(v[m].x, v[m].y);
      *reinterpret_cast<uint32_t*>(orow + 4 * i) = (*reinterpret_cast<const uint32_t*>(&bb)) ^ msk[m].x;
    } else {
      *reinterpret_cast<uint2*>(orow + 8 * i) =
          make_uint2(__float_as_uint(v[m].x) ^ msk[m].x, __float_as_uint(v[m].y) ^ msk[m].y);
    }
  }
}

template <int D, typename TOut>
__device__ __forceinline__ void store_out_tile(const DecJob& J, const uint8_t* smem, int row0, int nrows, int tid) {
  using C = Dec<D, TOut>;
  using OT = typename C::OT;
  uint8_t* y = reinterpret_cast<uint8_t*>(J.y);
#pragma unroll
  for (int q = 0; q < C::CHUNKS; ++q) {
    const int id = q * kThreads + tid;
    const int r = id / OT::CPR;
    const int c = id - r * OT::CPR;
    if (r < nrows) {
      const uint4 v = *reinterpret_cast<const uint4*>(smem + C::OFF_OUT + r * OT::STRIDE + c * 16);
      *reinterpret_cast<uint4*>(y + ((int64_t)(row0 + r) * J.stride) * C::ESZ + c * 16) = v;
    }
  }
}

template <int D, typename TOut>
__global__ void __launch_bounds__(kThreads, 3) decode_kernel(const __grid_constant__ DecParams p) {
  using C = Dec<D, TOut>;
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x;
  const int G = gridDim.x;
  int t = blockIdx.x;
  if (t >= p.ntiles) return;

  // Centre tables for every n = 2..256: (cos + sin, cos - sin)(2 pi k / n) / sqrt(d).
  float2* ttab = reinterpret_cast<float2*>(smem + C::OFF_TAB);
  const float sc = sqrtf(2.f / (float)D);  // sqrt2 / sqrt(d)
  for (int idx = tid; idx < kTabEntries - 2; idx += kThreads) {
    const int w = 31 - __clz(idx + 2);
    const int k = idx - tab_offset(w);
    const float2 cs = cos_sin_q8(centre_q8(k, 1 << w), 1 << w);  // (cos psi, sin psi), psi = phi + pi/4
    ttab[idx] = make_float2(sc * cs.y, sc * cs.x);
  }

  int jid = find_job(p, t);
  int mask_jid = -1;
  uint2 msk[8];
#pragma unroll
  for (int s = 0; s < kStages - 1; ++s) {
    const int ts = t + s * G;
    if (ts < p.ntiles) {
      const DecJob& Js = p.job[find_job(p, ts)];
      const int rs = (ts - Js.tile0) * C::TR;
      issue_rec_load<D, TOut>(Js, rs, (int)min((int64_t)C::TR, Js.rows - rs), smem + C::OFF_REC + s * C::REC_B, tid);
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
        const DecJob& Jn = p.job[find_job(p, tn)];
        const int rn = (tn - Jn.tile0) * C::TR;
        issue_rec_load<D, TOut>(Jn, rn, (int)min((int64_t)C::TR, Jn.rows - rn), smem + C::OFF_REC + nb * C::REC_B, tid);
      }
      cp_async_commit();
    }
    const DecJob& J = p.job[jid];
    if (jid != mask_jid) {
      const int l = tid % C::L;
#pragma unroll
      for (int m = 0; m < 8; ++m) msk[m] = pair_sign_mask<C::ESZ>(J.signs, l + C::L * m);
      mask_jid = jid;
    }
    const int row0 = (t - J.tile0) * C::TR;
    const int nrows = (int)min((int64_t)C::TR, J.rows - row0);
    const uint8_t* rec = smem + C::OFF_REC + cur * C::REC_B;

#define TAC_DEC_CASE(WW)                                                      \
  case WW:                                                                    \
    if (J.b == 8) decode_row<D, TOut, WW, 8>(J, rec, smem, tid, msk);         \
    else decode_row<D, TOut, WW, 4>(J, rec, smem, tid, msk);                  \
    break;
    switch (J.w) {
      TAC_DEC_CASE(1) TAC_DEC_CASE(2) TAC_DEC_CASE(3) TAC_DEC_CASE(4)
      TAC_DEC_CASE(5) TAC_DEC_CASE(6) TAC_DEC_CASE(7) TAC_DEC_CASE(8)
      default: break;
    }
#undef TAC_DEC_CASE
    __syncthreads();
    store_out_tile<D, TOut>(J, smem, row0, nrows, tid);

    if (t + G < p.ntiles) jid = find_job(p, t + G);
    cur = (cur + 1 == kStages) ? 0 : cur + 1;
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
