// Attention straight from TurboAngle records, for sm_103a.
//
// The consumer of the Sec. 3.1 reconstruction (the paper evaluates its codes
// through a model's attention but describes no kernel for it).  H and D are
// orthogonal and H is symmetric, so for a decoded key k^ = D H y^,
//   q . k^ = (H D q) . y^,      y^_2i + i y^_2i+1 = r^_i exp(2 pi i k_i / n),
// and the output sum_t p_t v^_t = D H (sum_t p_t y^V_t).  Scores are taken
// against the rotated query and values are accumulated in the rotated domain:
// one transform per query and one per output instead of one per cached token.
//
// Two kernels (flash-decoding split over tokens):
//   attend_partial  a CTA of 4 warps serves 4 consecutive splits of 256 tokens
//                   of one job.  The CTA rotates its queries once (fp32
//                   butterfly, times scale * log2 e for a base-2 softmax) and
//                   builds the K and V bin-centre tables (cos, sin)(2 pi k / n).
//                   Each warp streams its split in steps of RW tokens: a
//                   cp.async ring stages the six record segments (K and V
//                   angle / norm / header) of a step; K scores in the lane
//                   layout of the decoder (L lanes per token, 8 pairs per
//                   lane, shuffle reduction), an online softmax per query, V
//                   accumulated with lane l owning pairs l + 32 j.  Each warp
//                   writes (max, sum, accumulator) of its split to the workspace.
//   attend_combine  one warp per (job, query): merges the splits, divides,
//                   applies D H (fp32 butterfly) and stores the row.
// Codebooks (n, norm bits, norm mode) are runtime parameters: K and V may
// differ, and any codebook the encoder supports is accepted.
#include <atomic>

#include "tac_common.cuh"

namespace tac {

constexpr int kAttWarps = 4;                  // warps (splits) per CTA
constexpr int kAttThreads = 32 * kAttWarps;
constexpr int kAttSplit = TAC_ATTEND_SPLIT;   // tokens per split
constexpr int kAttNS = 3;                     // record stages per warp
constexpr float kLog2e = 1.4426950408889634f;

template <int D>
struct Att {
  using G = Geo<D>;
  static constexpr int P = G::P, L = G::L, RW = G::RW;
  static constexpr int PV = P / 32 > 0 ? P / 32 : 1;         // V pairs per lane (d = 64: 1, 128: 2)
  // record stage: K angle | K norm | K header | V angle | V norm | V header, each
  // at most RW * (P, 4P, 8) bytes (angle codes <= 8 bits, fp32 norms)
  static constexpr int SEG_A = RW * P, SEG_N = RW * 4 * P, SEG_H = RW * 8;
  static constexpr int S_KA = 0, S_KN = S_KA + SEG_A, S_KH = S_KN + SEG_N;
  static constexpr int S_VA = S_KH + SEG_H, S_VN = S_VA + SEG_A, S_VH = S_VN + SEG_N;
  static constexpr int STAGE = S_VH + SEG_H + 16;            // + slack for funnel reads
  static constexpr int QROW = P + P / 8;                      // skewed rotated-query row (float2 units)
  // CTA shared memory
  static constexpr int OFF_Q = 0;                                             // float2 [TAC_MAX_QUERIES][QROW]
  static constexpr int OFF_TK = OFF_Q + TAC_MAX_QUERIES * QROW * 8;           // float2 [256] K (cos, sin)
  static constexpr int OFF_TV = OFF_TK + 256 * 8;                             // float2 [256] V (cos, sin)
  static constexpr int OFF_W = OFF_TV + 256 * 8;                              // per-warp stages
  static constexpr int SMEM = OFF_W + kAttWarps * kAttNS * STAGE;
  static_assert(STAGE % 16 == 0 && OFF_W % 16 == 0, "alignment");
};

// The skewed position of pair i in a rotated-query row: pairs 8l..8l+7 of the
// L lanes of a row then fall on distinct bank pairs.
__device__ __forceinline__ int qpos(int i) { return i + (i >> 3); }

// Up to 8 bytes from a shared byte address with any alignment.
__device__ __forceinline__ uint64_t load_u64_any(const uint8_t* p) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  const uint32_t* w = reinterpret_cast<const uint32_t*>(a & ~(uintptr_t)3);
  const int sh = (int)(a & 3) * 8;
  const uint64_t lo = (uint64_t)w[0] | ((uint64_t)w[1] << 32);
  uint64_t v = lo >> sh;
  if (sh) v |= (uint64_t)w[2] << (64 - sh);
  return v;
}

// Dequantization constants of one record (the inverse of Eq. 2): r^ = base + c step
// (linear) or 2^(base + c step) (log); inv_l = 1 / (2^b - 1).
__device__ __forceinline__ float2 norm_consts(const uint8_t* hdr, float inv_l, int mode) {
  const float2 h = *reinterpret_cast<const float2*>(hdr);
  const bool spread = h.y > h.x;
  if (mode == TAC_NORM_LINEAR) return make_float2(h.x, spread ? (h.y - h.x) * inv_l : 0.f);
  const float lmin = lg2_approx(h.x);
  return make_float2(lmin, spread ? (lg2_approx(h.y) - lmin) * inv_l : 0.f);
}

__device__ __forceinline__ float dequant(uint32_t c, float2 bs, int mode) {
  const float v = __fmaf_rn((float)c, bs.y, bs.x);
  return mode == TAC_NORM_LOG ? ex2_approx(v) : v;
}

// In-place normalized Walsh-Hadamard transform of `rows` rows of d floats in
// shared memory (Sylvester order), by the nthreads threads of the caller.
template <int D>
__device__ __forceinline__ void smem_fwht(float* buf, int rows, int tid, int nthreads, bool block_sync) {
  for (int h = 1; h < D; h <<= 1) {
    if (block_sync) __syncthreads(); else __syncwarp();
    for (int e = tid; e < rows * D / 2; e += nthreads) {
      const int r = e / (D / 2), k = e % (D / 2);
      const int i = (k / h) * 2 * h + (k % h);
      float* row = buf + r * D;
      const float a = row[i], b = row[i + h];
      row[i] = a + b;
      row[i + h] = a - b;
    }
  }
  if (block_sync) __syncthreads(); else __syncwarp();
}

template <int D, typename TQ, int NQ>
__global__ void __launch_bounds__(kAttThreads) attend_partial(const __grid_constant__ AttParams p, float* ws) {
  using C = Att<D>;
  using G = Geo<D>;
  constexpr int P = C::P, L = C::L, RW = C::RW, PV = C::PV;
  constexpr int ESZ = (int)sizeof(TQ);
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // ---- the CTA's job ----
  int jb = 0;
  {
    int lo = 0, hi = p.njobs - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (p.job[mid].cta0 <= (int)blockIdx.x) lo = mid; else hi = mid - 1;
    }
    jb = lo;
  }
  const AttJob& J = p.job[jb];
  const int nq = J.nq;

  // ---- rotated queries q' = H D_K q * scale * log2(e), skewed float2 rows ----
  float* qbuf = reinterpret_cast<float*>(smem + C::OFF_W);   // staging, reused by the record ring below
  for (int e = tid; e < nq * D; e += kAttThreads) {
    const int a = e / D, j = e % D;
    const uint8_t* qr = reinterpret_cast<const uint8_t*>(J.q) + (int64_t)a * J.q_stride * ESZ;
    float x;
    if constexpr (ESZ == 2) x = __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(qr)[j]);
    else x = reinterpret_cast<const float*>(qr)[j];
    qbuf[e] = ((J.sk[j >> 5] >> (j & 31)) & 1u) ? -x : x;
  }
  smem_fwht<D>(qbuf, nq, tid, kAttThreads, true);
  float2* qrot = reinterpret_cast<float2*>(smem + C::OFF_Q);
  const float qs = J.scale * kLog2e * rsqrtf((float)D);
  for (int e = tid; e < nq * P; e += kAttThreads) {
    const int a = e / P, i = e % P;
    qrot[a * C::QROW + qpos(i)] = make_float2(qbuf[a * D + 2 * i] * qs, qbuf[a * D + 2 * i + 1] * qs);
  }
  // ---- bin-centre tables (cos, sin)(2 pi k / n) ----
  float2* tk = reinterpret_cast<float2*>(smem + C::OFF_TK);
  float2* tv = reinterpret_cast<float2*>(smem + C::OFF_TV);
  for (int k = tid; k < J.nk; k += kAttThreads) tk[k] = cos_sin_q8(8 * k, J.nk);
  for (int k = tid; k < J.nv; k += kAttThreads) tv[k] = cos_sin_q8(8 * k, J.nv);
  __syncthreads();

  // ---- this warp's split ----
  const int split = J.split0 + ((int)blockIdx.x - J.cta0) * kAttWarps + warp;
  const int64_t t_begin = (int64_t)(split - J.split0) * kAttSplit;
  if (t_begin >= J.tokens) return;
  const int64_t t_stop = min(J.tokens, t_begin + kAttSplit);
  const int nsteps = (int)((t_stop - t_begin + RW - 1) / RW);
  uint8_t* wsm = smem + C::OFF_W + warp * kAttNS * C::STAGE;

  const int ak = P * J.wk / 8, nbk = P * J.bk / 8;     // K record bytes per row (angle, norm)
  const int av = P * J.wv / 8, nbv = P * J.bv / 8;
  const bool hk = J.mk != TAC_NORM_FP32, hv = J.mv != TAC_NORM_FP32;

  // Stage the records of step s (tokens t_begin + s*RW ...): six segments,
  // 16-byte chunks, bytes past the last token zero-filled.
  auto issue = [&](int s) {
    if (s < nsteps) {
      const int64_t row0 = t_begin + (int64_t)s * RW;
      const int rows = (int)min((int64_t)RW, J.tokens - row0);
      uint8_t* st = wsm + (s % kAttNS) * C::STAGE;
      const uint8_t* src[6] = {J.kc + row0 * ak, J.kn + row0 * nbk, J.kh + row0 * 8,
                               J.vc + row0 * av, J.vn + row0 * nbv, J.vh + row0 * 8};
      const int rb[6] = {ak, nbk, hk ? 8 : 0, av, nbv, hv ? 8 : 0};
      const int off[6] = {C::S_KA, C::S_KN, C::S_KH, C::S_VA, C::S_VN, C::S_VH};
#pragma unroll
      for (int g = 0; g < 6; ++g) {
        const int full = RW * rb[g], valid = rows * rb[g];
        for (int c = lane * 16; c < full; c += 32 * 16) {
          const int rem = valid - c;
          const int n = rem >= 16 ? 16 : (rem > 0 ? rem : 0);
          cp_async16(st + off[g] + c, n > 0 ? src[g] + c : src[g], n);
        }
      }
    }
    cp_async_commit();
  };
#pragma unroll
  for (int s = 0; s < kAttNS - 1; ++s) issue(s);

  const int r = lane / L, l = lane % L;     // K layout: token r of the step, pairs 8l..8l+7
  // V layout: lane owns pairs lane + 32 j; their code positions are fixed per job
  int va_w[PV], va_s[PV], vn_w[PV], vn_s[PV];
#pragma unroll
  for (int j = 0; j < PV; ++j) {
    const int i = lane + 32 * j, ba = i * J.wv, bn = i * J.bv;
    va_w[j] = ba >> 5; va_s[j] = ba & 31;
    vn_w[j] = bn >> 5; vn_s[j] = bn & 31;
  }
  const uint32_t vmask = (1u << J.wv) - 1u;
  const uint32_t nvmask = J.bv >= 32 ? 0xffffffffu : (1u << J.bv) - 1u;
  float m_run[NQ], l_run[NQ];
  float acc[NQ][PV][2];
#pragma unroll
  for (int a = 0; a < NQ; ++a) {
    m_run[a] = -INFINITY;
    l_run[a] = 0.f;
#pragma unroll
    for (int j = 0; j < PV; ++j) acc[a][j][0] = acc[a][j][1] = 0.f;
  }

  for (int s = 0; s < nsteps; ++s) {
    cp_async_wait<kAttNS - 2>();
    __syncwarp();
    issue(s + kAttNS - 1);
    const uint8_t* st = wsm + (s % kAttNS) * C::STAGE;
    const int64_t row0 = t_begin + (int64_t)s * RW;
    const int valid = (int)min((int64_t)RW, t_stop - row0);   // tokens of this step
    // dequantization constants of the V record of token r (broadcast in the V phase)
    const float2 vbs = hv ? norm_consts(st + C::S_VH + r * 8, J.inv_lv, J.mv) : make_float2(0.f, 0.f);

    // ---- K: partial scores of token r over pairs 8l..8l+7 ----
    float sc[NQ];
#pragma unroll
    for (int a = 0; a < NQ; ++a) sc[a] = 0.f;
    {
      const uint64_t ka = load_u64_any(st + C::S_KA + r * ak + l * J.wk);
      const uint32_t kmask = (1u << J.wk) - 1u;
      const float2 bs = hk ? norm_consts(st + C::S_KH + r * 8, J.inv_lk, J.mk) : make_float2(0.f, 0.f);
      const uint8_t* nrow = st + C::S_KN + r * nbk;
      uint64_t kn = 0;
      if (J.mk != TAC_NORM_FP32)
        kn = J.bk == 8 ? load_u64_any(nrow + l * 8) : (uint64_t)reinterpret_cast<const uint32_t*>(nrow)[l];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        uint32_t k = (uint32_t)(ka >> (j * J.wk)) & kmask;
        k = min(k, (uint32_t)(J.nk - 1));
        float rh;
        if (J.mk == TAC_NORM_FP32) rh = reinterpret_cast<const float*>(nrow)[8 * l + j];
        else rh = dequant((uint32_t)(kn >> (j * J.bk)) & ((1u << J.bk) - 1u), bs, J.mk);
        const float2 cs = tk[k];
        const float rc = rh * cs.x, rs = rh * cs.y;
        const int qi = qpos(8 * l + j);
#pragma unroll
        for (int a = 0; a < NQ; ++a) {
          if (a < nq) {
            const float2 qq = qrot[a * C::QROW + qi];
            sc[a] = __fmaf_rn(qq.x, rc, __fmaf_rn(qq.y, rs, sc[a]));
          }
        }
      }
    }
#pragma unroll
    for (int a = 0; a < NQ; ++a) {
      if (a < nq) {
#pragma unroll
        for (int off = 1; off < L; off <<= 1) sc[a] += __shfl_xor_sync(0xffffffffu, sc[a], off);
      }
    }

    // ---- online softmax over the step's tokens (base 2) ----
    float pw[NQ][RW];
#pragma unroll
    for (int a = 0; a < NQ; ++a) {
      if (a < nq) {
        float mx = m_run[a];
#pragma unroll
        for (int rr = 0; rr < RW; ++rr) {
          float v = __shfl_sync(0xffffffffu, sc[a], rr * L);
          if (rr >= valid) v = -INFINITY;
          pw[a][rr] = v;
          mx = fmaxf(mx, v);
        }
        const float f = ex2_approx(m_run[a] - mx);   // m_run = -inf at first: f = 0
        float sum = 0.f;
#pragma unroll
        for (int rr = 0; rr < RW; ++rr) {
          pw[a][rr] = ex2_approx(pw[a][rr] - mx);
          sum += pw[a][rr];
        }
        l_run[a] = __fmaf_rn(l_run[a], f, sum);
        m_run[a] = mx;
#pragma unroll
        for (int j = 0; j < PV; ++j) { acc[a][j][0] *= f; acc[a][j][1] *= f; }
      }
    }

    // ---- V: accumulate p_t y^V_t, lane l owning pairs l + 32 j ----
#pragma unroll
    for (int rr = 0; rr < RW; ++rr) {
      if (rr >= valid) break;
      const uint32_t* arow = reinterpret_cast<const uint32_t*>(st + C::S_VA + rr * av);
      const uint32_t* nrow = reinterpret_cast<const uint32_t*>(st + C::S_VN + rr * nbv);
      const float2 bs = make_float2(__shfl_sync(0xffffffffu, vbs.x, rr * L), __shfl_sync(0xffffffffu, vbs.y, rr * L));
#pragma unroll
      for (int j = 0; j < PV; ++j) {
        const int i = lane + 32 * j;
        if (i < P) {
          uint32_t k = __funnelshift_r(arow[va_w[j]], arow[va_w[j] + 1], va_s[j]) & vmask;
          k = min(k, (uint32_t)(J.nv - 1));
          float rh;
          if (J.mv == TAC_NORM_FP32) rh = __uint_as_float(nrow[i]);
          else rh = dequant((nrow[vn_w[j]] >> vn_s[j]) & nvmask, bs, J.mv);
          const float2 cs = tv[k];
          const float yc = rh * cs.x, ys = rh * cs.y;
#pragma unroll
          for (int a = 0; a < NQ; ++a) {
            if (a < nq) {
              acc[a][j][0] = __fmaf_rn(pw[a][rr], yc, acc[a][j][0]);
              acc[a][j][1] = __fmaf_rn(pw[a][rr], ys, acc[a][j][1]);
            }
          }
        }
      }
    }
  }
  cp_async_wait<0>();

  // ---- write the split's partial results ----
  float* rec = ws + J.ws + (int64_t)(split - J.split0) * nq * att_rec_floats(D);
#pragma unroll
  for (int a = 0; a < NQ; ++a) {
    if (a < nq) {
      float* ra = rec + a * att_rec_floats(D);
      if (lane == 0) { ra[0] = m_run[a]; ra[1] = l_run[a]; }
#pragma unroll
      for (int j = 0; j < PV; ++j) {
        const int i = lane + 32 * j;
        if (i < P) *reinterpret_cast<float2*>(ra + 2 + 2 * i) = make_float2(acc[a][j][0], acc[a][j][1]);
      }
    }
  }
}

// One warp per (job, query): merge the splits, normalize, out = D_V H y.
template <int D, typename TO>
__global__ void __launch_bounds__(128) attend_combine(const __grid_constant__ AttParams p, const float* ws,
                                                      int nrows_total) {
  constexpr int ESZ = (int)sizeof(TO);
  __shared__ float buf[4][D];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = blockIdx.x * 4 + warp;           // global (job, query) index
  if (g >= nrows_total) return;
  int jb = 0, base = 0;
  for (; jb < p.njobs; ++jb) {
    if (g < base + p.job[jb].nq) break;
    base += p.job[jb].nq;
  }
  const AttJob& J = p.job[jb];
  const int a = g - base;
  const int nsp = (int)((J.tokens + kAttSplit - 1) / kAttSplit);
  const float* recs = ws + J.ws;
  float M = -INFINITY;
  for (int s = 0; s < nsp; ++s) M = fmaxf(M, recs[((int64_t)s * J.nq + a) * att_rec_floats(D)]);
  float Lsum = 0.f;
  float y[D / 32];
#pragma unroll
  for (int e = 0; e < D / 32; ++e) y[e] = 0.f;
  for (int s = 0; s < nsp; ++s) {
    const float* ra = recs + ((int64_t)s * J.nq + a) * att_rec_floats(D);
    const float f = ex2_approx(ra[0] - M);
    Lsum = __fmaf_rn(ra[1], f, Lsum);
#pragma unroll
    for (int e = 0; e < D / 32; ++e) y[e] = __fmaf_rn(ra[2 + lane + 32 * e], f, y[e]);
  }
  const float inv = 1.f / Lsum;
  float* row = buf[warp];
#pragma unroll
  for (int e = 0; e < D / 32; ++e) row[lane + 32 * e] = y[e] * inv;
  smem_fwht<D>(row, 1, lane, 32, false);
  const float sc = rsqrtf((float)D);
  uint8_t* orow = reinterpret_cast<uint8_t*>(J.out) + (int64_t)a * J.out_stride * ESZ;
#pragma unroll
  for (int e = 0; e < D / 32; ++e) {
    const int j = lane + 32 * e;
    float v = row[j] * sc;
    if ((J.sv[j >> 5] >> (j & 31)) & 1u) v = -v;
    if constexpr (ESZ == 2) reinterpret_cast<__nv_bfloat16*>(orow)[j] = __float2bfloat16_rn(v);
    else reinterpret_cast<float*>(orow)[j] = v;
  }
}

template <int D, typename TQ, int NQ>
static cudaError_t launch_attend_t(const AttParams& p, int nrows_total, float* ws, cudaStream_t st) {
  using C = Att<D>;
  auto kp = attend_partial<D, TQ, NQ>;
  static int configured[64] = {0};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kp, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    configured[dev] = 1;
  }
  if (p.nctas > 0) kp<<<p.nctas, kAttThreads, C::SMEM, st>>>(p, ws);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int blocks = (nrows_total + 3) / 4;
  if (blocks > 0) attend_combine<D, TQ><<<blocks, 128, 0, st>>>(p, ws, nrows_total);
  return cudaGetLastError();
}

// The workspace of tac_attend_multi_static: one array per device, in the
// module image (no allocation at call time).
static __device__ __align__(256) float g_attend_ws[TAC_ATTEND_STATIC_WS_BYTES / 4];

// Address of g_attend_ws on the current device, resolved once per device.
cudaError_t attend_static_workspace(float** ws) {
  constexpr int kMaxDevices = 64;
  static std::atomic<void*> cache[kMaxDevices];
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  void* a = cache[dev].load(std::memory_order_acquire);
  if (!a) {
    e = cudaGetSymbolAddress(&a, g_attend_ws);
    if (e != cudaSuccess) return e;
    if (!a || (reinterpret_cast<uintptr_t>(a) & 255)) return cudaErrorInvalidSymbol;
    cache[dev].store(a, std::memory_order_release);   // racing first calls store the same address
  }
  *ws = static_cast<float*>(a);
  return cudaSuccess;
}

// nq_max: the largest query count of the jobs (the kernel is built for 1, 2, 4, 8).
cudaError_t launch_attend(int d, int dtype, int nq_max, const AttParams& p, int nrows_total, float* ws,
                          cudaStream_t st) {
  const bool bf = dtype == TAC_BF16;
#define TAC_ATT_NQ(DD, T)                                                           \
  if (nq_max <= 1) return launch_attend_t<DD, T, 1>(p, nrows_total, ws, st);        \
  if (nq_max <= 2) return launch_attend_t<DD, T, 2>(p, nrows_total, ws, st);        \
  if (nq_max <= 4) return launch_attend_t<DD, T, 4>(p, nrows_total, ws, st);        \
  return launch_attend_t<DD, T, 8>(p, nrows_total, ws, st);
  if (d == 64) { if (bf) { TAC_ATT_NQ(64, __nv_bfloat16) } else { TAC_ATT_NQ(64, float) } }
  if (d == 128) { if (bf) { TAC_ATT_NQ(128, __nv_bfloat16) } else { TAC_ATT_NQ(128, float) } }
#undef TAC_ATT_NQ
  return cudaErrorInvalidValue;
}

}  // namespace tac
