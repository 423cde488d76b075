// TurboAngle decode kernel for sm_103a (Sec. 3.1 reconstruction with the Eq. 2
// dequantization of arXiv 2603.27467).
//
// One thread owns one row of a 128-row tile:
//   1. the tile's records (angle / norm / header planes) are staged global ->
//      shared with cp.async: coalesced 16-byte chunks for contiguous slots,
//      per-row copies for gathered slots; double buffered;
//   2. each pair is rebuilt from its bin-centre angle by table lookup: the table
//      holds (cos phi_k + sin phi_k, cos phi_k - sin phi_k) / sqrt(d), i.e. the
//      element-pair butterfly stage and the 1/sqrt(d) normalization are folded
//      into the lookup, so the remaining log2(d) - 1 butterfly stages run on
//      packed fp32 pairs (FADD2/FFMA2) straight from (E_i, O_i) = r^_i * T[k_i];
//   3. D is applied as a sign XOR on the output bits (after bf16 RNE rounding,
//      or on fp32), rows are staged swizzled and written with coalesced stores.
#include "tac_common.cuh"

namespace tac {

template <int D, typename TOut>
struct Dec {
  static constexpr int P = D / 2;
  static constexpr int ESZ = (int)sizeof(TOut);
  static constexpr int ROWB = D * ESZ;                 // output row bytes
  static constexpr int CPR = ROWB / 16;
  static constexpr int ABMAX = P;                      // angle record bytes at w = 8
  static constexpr int NBMAX = P;                      // norm record bytes at b = 8
  static constexpr int REC_B = kTileRows * (ABMAX + NBMAX + 8);  // one record buffer
  // shared memory layout (bytes)
  static constexpr int OFF_REC = 0;                    // 2 record buffers
  static constexpr int OFF_OUT = OFF_REC + 2 * REC_B;  // output tile
  static constexpr int OFF_TAB = OFF_OUT + kTileRows * ROWB;
  static constexpr int OFF_MSK = OFF_TAB + kTabEntries * 8;
  static constexpr int SMEM = OFF_MSK + P * 8;
  // inside a record buffer
  static constexpr int R_ANG = 0;
  static constexpr int R_NRM = kTileRows * ABMAX;
  static constexpr int R_HDR = R_NRM + kTileRows * NBMAX;
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
  const int P = C::P;
  const int AB = P * J.w / 8, NB = P * J.b / 8;
  if (J.slot == nullptr) {
    cta_copy_in(buf + C::R_ANG, J.codes + (int64_t)row0 * AB, nrows * AB, tid);
    cta_copy_in(buf + C::R_NRM, J.norms + (int64_t)row0 * NB, nrows * NB, tid);
    cta_copy_in(buf + C::R_HDR, J.hdr + (int64_t)row0 * 8, nrows * 8, tid);
  } else if (tid < nrows) {
    // Gather: this thread's record, byte-exact, with plain loads (records of odd
    // size are not 16-byte aligned in the source planes).
    int64_t s = J.slot[row0 + tid];
    uint8_t* da = buf + C::R_ANG + tid * AB;
    uint8_t* dn = buf + C::R_NRM + tid * NB;
    float2* dh = reinterpret_cast<float2*>(buf + C::R_HDR) + tid;
    if (s < 0 || s >= J.capacity) {  // out-of-range slot: decodes as an all-zero record
      for (int q = 0; q < AB; ++q) da[q] = 0;
      for (int q = 0; q < NB; ++q) dn[q] = 0;
      *dh = make_float2(0.f, 0.f);
      return;
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

template <int D, typename TOut>
__device__ __forceinline__ void build_dec_masks(const DecJob& J, uint2* msk, int tid) {
  using C = Dec<D, TOut>;
  for (int i = tid; i < C::P; i += kThreads) {
    const uint32_t b0 = (J.signs[(2 * i) >> 5] >> ((2 * i) & 31)) & 1u;
    const uint32_t b1 = (J.signs[(2 * i + 1) >> 5] >> ((2 * i + 1) & 31)) & 1u;
    if constexpr (C::ESZ == 2) msk[i] = make_uint2((b0 << 15) | (b1 << 31), 0u);
    else msk[i] = make_uint2(b0 << 31, b1 << 31);
  }
}

// Read W bits at bit offset `bit` of a little-endian word array (compile-time offsets).
template <int W>
__device__ __forceinline__ uint32_t get_bits(const uint32_t* a, int bit) {
  const int wi = bit >> 5, sh = bit & 31;
  uint32_t v = a[wi] >> sh;
  if (sh + W > 32) v |= a[wi + 1] << (32 - sh);
  return v & ((1u << W) - 1u);
}

template <int BYTES, int NWORDS>
__device__ __forceinline__ void load_record(uint32_t (&w)[NWORDS], const uint8_t* src) {
  if constexpr (BYTES % 16 == 0) {
#pragma unroll
    for (int q = 0; q < BYTES / 16; ++q) {
      const uint4 t = reinterpret_cast<const uint4*>(src)[q];
      w[4 * q] = t.x; w[4 * q + 1] = t.y; w[4 * q + 2] = t.z; w[4 * q + 3] = t.w;
    }
  } else if constexpr (BYTES % 8 == 0) {
#pragma unroll
    for (int q = 0; q < BYTES / 8; ++q) {
      const uint2 t = reinterpret_cast<const uint2*>(src)[q];
      w[2 * q] = t.x; w[2 * q + 1] = t.y;
    }
  } else if constexpr (BYTES % 4 == 0) {
#pragma unroll
    for (int q = 0; q < BYTES / 4; ++q) w[q] = reinterpret_cast<const uint32_t*>(src)[q];
  } else {
#pragma unroll
    for (int q = 0; q < NWORDS; ++q) w[q] = 0u;
#pragma unroll
    for (int q = 0; q < BYTES; ++q) w[q >> 2] |= (uint32_t)src[q] << (8 * (q & 3));
  }
}

template <int D, typename TOut, int W, int B>
__device__ __forceinline__ void decode_row(const DecJob& J, const uint8_t* rec, uint8_t* smem, int tid) {
  using C = Dec<D, TOut>;
  constexpr int P = C::P;
  constexpr int AB = P * W / 8;
  constexpr int NB = P * B / 8;
  constexpr int AW = (P * W + 31) / 32;
  constexpr int NW = (P * B + 31) / 32;
  constexpr int L = (1 << B) - 1;
  const float2* ttab = reinterpret_cast<const float2*>(smem + C::OFF_TAB) + tab_offset(W);
  const uint2* msk = reinterpret_cast<const uint2*>(smem + C::OFF_MSK);

  uint32_t aw[AW], nw[NW];
  load_record<AB>(aw, rec + C::R_ANG + tid * AB);
  load_record<NB>(nw, rec + C::R_NRM + tid * NB);
  const float2 h = reinterpret_cast<const float2*>(rec + C::R_HDR)[tid];
  const float hmin = h.x, hmax = h.y;

  // Dequantization (reading of Eq. 2's inverse): linear r^ = r_min + c (r_max - r_min)/L,
  // log r^ = 2^(l_min + c (l_max - l_min)/L); r_max == r_min gives r^ = r_min.
  const bool flat = !(hmax != hmin);
  float base, step;
  if (J.mode == TAC_NORM_LINEAR) {
    base = hmin;
    step = __fdiv_rn(__fsub_rn(hmax, hmin), (float)L);
  } else {
    base = flat ? 0.f : log2f(hmin);
    step = flat ? 0.f : __fdiv_rn(__fsub_rn(log2f(hmax), base), (float)L);
  }

  float2 v[P];
#pragma unroll
  for (int i = 0; i < P; ++i) {
    const uint32_t k = get_bits<W>(aw, i * W);
    const uint32_t c = get_bits<B>(nw, i * B);
    float r;
    if (J.mode == TAC_NORM_LINEAR) r = __fmaf_rn((float)c, step, base);
    else r = exp2f(__fmaf_rn((float)c, step, base));
    if (flat) r = hmin;
    const float2 t = ttab[k];
    v[i] = mul2(make_float2(r, r), t);
  }
  // Remaining butterfly stages (input bits 1..log2 d - 1); H is its own inverse (Sec. 2).
#pragma unroll
  for (int hh = 1; hh < P; hh <<= 1) {
#pragma unroll
    for (int i = 0; i < P; ++i) {
      if ((i & hh) == 0) {
        const float2 a = v[i], b = v[i + hh];
        v[i] = add2(a, b);
        v[i + hh] = sub2(a, b);
      }
    }
  }
  // D, convert, stage the row (swizzled).
  uint8_t* orow = smem + C::OFF_OUT + tid * C::ROWB;
  const int sw = row_swz<C::ROWB>(tid);
  if constexpr (C::ESZ == 2) {
#pragma unroll
    for (int c = 0; c < C::CPR; ++c) {
      uint32_t q[4];
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int i = 4 * c + t;
        const __nv_bfloat162 b = __floats2bfloat162_rn(v[i].x, v[i].y);
        q[t] = (*reinterpret_cast<const uint32_t*>(&b)) ^ msk[i].x;
      }
      *reinterpret_cast<uint4*>(orow + ((c ^ sw) << 4)) = make_uint4(q[0], q[1], q[2], q[3]);
    }
  } else {
#pragma unroll
    for (int c = 0; c < C::CPR; ++c) {
      const int i0 = 2 * c, i1 = 2 * c + 1;
      *reinterpret_cast<uint4*>(orow + ((c ^ sw) << 4)) =
          make_uint4(__float_as_uint(v[i0].x) ^ msk[i0].x, __float_as_uint(v[i0].y) ^ msk[i0].y,
                     __float_as_uint(v[i1].x) ^ msk[i1].x, __float_as_uint(v[i1].y) ^ msk[i1].y);
    }
  }
}

template <int D, typename TOut>
__device__ __forceinline__ void store_out_tile(const DecJob& J, const uint8_t* smem, int row0, int nrows, int tid) {
  using C = Dec<D, TOut>;
  uint8_t* y = reinterpret_cast<uint8_t*>(J.y);
  const int total = nrows * C::CPR;
  for (int id = tid; id < total; id += kThreads) {
    const int r = id / C::CPR;
    const int c = id - r * C::CPR;
    const uint4 q = *reinterpret_cast<const uint4*>(smem + C::OFF_OUT + r * C::ROWB + ((c ^ row_swz<C::ROWB>(r)) << 4));
    *reinterpret_cast<uint4*>(y + ((int64_t)(row0 + r) * J.stride) * C::ESZ + c * 16) = q;
  }
}

template <int D, typename TOut>
__global__ void __launch_bounds__(kThreads, 2) decode_kernel(const __grid_constant__ DecParams p) {
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
  build_dec_masks<D, TOut>(p.job[jid], reinterpret_cast<uint2*>(smem + C::OFF_MSK), tid);
  {
    const DecJob& J = p.job[jid];
    const int row0 = (t - J.tile0) * kTileRows;
    issue_rec_load<D, TOut>(J, row0, (int)min((int64_t)kTileRows, J.rows - row0), smem + C::OFF_REC, tid);
    cp_async_commit();
    const int t1 = t + G;
    if (t1 < p.ntiles) {
      const DecJob& J1 = p.job[find_job(p, t1)];
      const int r1 = (t1 - J1.tile0) * kTileRows;
      issue_rec_load<D, TOut>(J1, r1, (int)min((int64_t)kTileRows, J1.rows - r1), smem + C::OFF_REC + C::REC_B, tid);
    }
    cp_async_commit();
  }

  int cur = 0;
  for (; t < p.ntiles; t += G) {
    cp_async_wait<1>();
    __syncthreads();
    const DecJob& J = p.job[jid];
    const int row0 = (t - J.tile0) * kTileRows;
    const int nrows = (int)min((int64_t)kTileRows, J.rows - row0);
    const uint8_t* rec = smem + C::OFF_REC + cur * C::REC_B;

#define TAC_DEC_CASE(WW)                                                      \
  case WW:                                                                    \
    if (J.b == 8) decode_row<D, TOut, WW, 8>(J, rec, smem, tid);              \
    else decode_row<D, TOut, WW, 4>(J, rec, smem, tid);                       \
    break;
    switch (J.w) {
      TAC_DEC_CASE(1) TAC_DEC_CASE(2) TAC_DEC_CASE(3) TAC_DEC_CASE(4)
      TAC_DEC_CASE(5) TAC_DEC_CASE(6) TAC_DEC_CASE(7) TAC_DEC_CASE(8)
      default: break;
    }
#undef TAC_DEC_CASE
    __syncthreads();
    store_out_tile<D, TOut>(J, smem, row0, nrows, tid);

    const int t2 = t + 2 * G;
    if (t2 < p.ntiles) {
      const DecJob& J2 = p.job[find_job(p, t2)];
      const int r2 = (t2 - J2.tile0) * kTileRows;
      issue_rec_load<D, TOut>(J2, r2, (int)min((int64_t)kTileRows, J2.rows - r2), smem + C::OFF_REC + cur * C::REC_B, tid);
    }
    cp_async_commit();
    if (t + G < p.ntiles) {
      jid = find_job(p, t + G);
      build_dec_masks<D, TOut>(p.job[jid], reinterpret_cast<uint2*>(smem + C::OFF_MSK), tid);
    }
    cur ^= 1;
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
