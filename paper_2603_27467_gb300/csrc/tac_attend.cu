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
#include <algorithm>
#include <atomic>

#include "tac_attend.cuh"

namespace tac {

template <int V>
struct IC { static constexpr int value = V; };

constexpr int kAttMaxWarps = 6;               // warps (splits) per CTA: 1..6, chosen per launch
constexpr int kAttSplit = TAC_ATTEND_SPLIT;   // tokens per split (one warp)
constexpr int kAttNS = 2;                     // staged batches per warp
constexpr float kLog2e = 1.4426950408889634f;
static_assert(kAttSplit % kAttBatch == 0, "a split is whole batches");

template <int D, int NQ>
struct Att {
  using G = Geo<D>;
  static constexpr int P = G::P, L = G::L, RW = G::RW;   // K: L lanes per token, RW tokens per pass
  static constexpr int PV = P / 32;                      // V: pairs per lane
  static constexpr int QROW = P + P / 4;                 // skewed rotated-query row (float2 units)
  static constexpr int PBROW = 16 + 16 * ((NQ + 1) / 2); // per token: V constants, then (p, p) per query
  static constexpr int PB = kAttBatch * PBROW;
  // CTA shared memory: rotated queries | K table | V table | per warp (PB, kAttNS stages)
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_TK = OFF_Q + NQ * QROW * 8;
  static constexpr int OFF_TV = OFF_TK + kAttTabBytes;
  static constexpr int OFF_W = OFF_TV + kAttTabBytes;
  static constexpr int smem(int stage, int warps) { return OFF_W + warps * (PB + kAttNS * stage); }
  static_assert(OFF_TK % 16 == 0 && PB % 16 == 0 && P % 32 == 0, "layout");
};

// The skewed position of pair i in a rotated-query row: the 16-byte granules
// (pairs 8l + 2m, 8l + 2m + 1) of the L lanes of a token fall on distinct banks.
__device__ __forceinline__ int qpos(int i) { return i + 2 * (i >> 3); }

__device__ __forceinline__ uint32_t rotr(uint32_t x, int s) { return __funnelshift_r(x, x, s); }

// A shared-memory float4 load the compiler may not hoist or merge: keeps a
// loop-invariant operand in shared memory instead of in registers.
__device__ __forceinline__ float4 lds_f4_reload(const void* ptr) {
  float4 v;
  const uint32_t a = (uint32_t)__cvta_generic_to_shared(ptr);
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];\n" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(a));
  return v;
}

// Reduce-scatter over the L lanes of a token, as a tree over the passes: the
// lane's value for the pass set {I + k S} is its half, selected by lane bit S,
// of the two sets {I + 2kS} and {I + S + 2kS}, plus the partner's.  At the
// top (I = 0, S = 1) lane l holds the sum over the L lanes of pass l.  The
// two passes of a base set {I, I + L/2} are computed together (one call).
template <int L, int I, int S, int NQ, typename PF>
__device__ __forceinline__ void att_tree(PF& pass, int l, float (&v)[NQ]) {
  float va[NQ], vb[NQ];
  if constexpr (2 * S == L) {
    pass(IC<I>{}, IC<I + S>{}, va, vb);
  } else {
    att_tree<L, I, 2 * S, NQ>(pass, l, va);
    att_tree<L, I + S, 2 * S, NQ>(pass, l, vb);
  }
  const bool up = (l & S) != 0;
#pragma unroll
  for (int a = 0; a < NQ; ++a) {
    const float kept = up ? vb[a] : va[a];
    const float send = up ? va[a] : vb[a];
    v[a] = kept + __shfl_xor_sync(0xffffffffu, send, S);
  }
}

// (A, B) of one record's norms: r^ = A f + B for the code c entered as
// f = 1 + c 2^-b (its bits in the mantissa of 1.0); log mode gives log2 r^.
// This is the inverse of Eq. 2: base + c step = f 2^b step + (base - 2^b step).
__device__ __forceinline__ float2 norm_ab(float2 h, float inv_l, float two_b, bool lg) {
  const float lo = lg ? lg2_approx(h.x) : h.x;
  const float hi = lg ? lg2_approx(h.y) : h.y;
  const float step = h.y > h.x ? (hi - lo) * inv_l : 0.f;
  const float A = step * two_b;
  return make_float2(A, lo - A);
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

template <int D, int NQ>
__global__ void __launch_bounds__(32 * kAttMaxWarps, NQ <= 4 ? 2 : 1) attend_partial(const __grid_constant__ AttParams p, float* ws) {
  using C = Att<D, NQ>;
  constexpr int P = C::P, L = C::L, RW = C::RW, PV = C::PV;
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nthr = blockDim.x, wpc = nthr >> 5;

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

  // ---- batch geometry of this job's records ----
  const int ak = P * J.wk / 8, nbk = P * J.bk / 8, av = P * J.wv / 8, nbv = P * J.bv / 8;
  const int hkb = J.mk != TAC_NORM_FP32 ? 8 : 0, hvb = J.mv != TAC_NORM_FP32 ? 8 : 0;
  const int S_KN = kAttBatch * ak, S_KH = S_KN + kAttBatch * nbk, S_VA = S_KH + kAttBatch * hkb;
  const int S_VN = S_VA + kAttBatch * av, S_VH = S_VN + kAttBatch * nbv;
  const int stage = S_VH + kAttBatch * hvb + 16;   // == att_stage_bytes(...)

  // ---- rotated queries q' = H D_K q * scale * log2(e), skewed float2 rows ----
  float* qbuf = reinterpret_cast<float*>(smem + C::OFF_W);   // staging, reused by the batches below
  for (int e = tid; e < nq * D; e += nthr) {
    const int a = e / D, j = e % D;
    float x;
    if (p.q_bf16) {
      x = __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(J.q)[(int64_t)a * J.q_stride + j]);
    } else {
      x = reinterpret_cast<const float*>(J.q)[(int64_t)a * J.q_stride + j];
    }
    qbuf[e] = ((J.sk[j >> 5] >> (j & 31)) & 1u) ? -x : x;
  }
  smem_fwht<D>(qbuf, nq, tid, nthr, true);
  float2* qrot = reinterpret_cast<float2*>(smem + C::OFF_Q);
  const float qs = J.scale * kLog2e * rsqrtf((float)D);
  for (int e = tid; e < NQ * P; e += nthr) {   // in record (slot) order: slot i holds pair slot_pair(i)
    const int a = e / P, i = e % P, ip = slot_pair<D>(i);
    qrot[a * C::QROW + qpos(i)] =
        a < nq ? make_float2(qbuf[a * D + 2 * ip] * qs, qbuf[a * D + 2 * ip + 1] * qs) : make_float2(0.f, 0.f);
  }
  // ---- bin-centre tables (cos, sin)(2 pi k / n), 2^lgr copies: entry k copy c
  // at k 2^lgr + c; entries n..2^W-1 repeat entry n-1 (codes >= n clamp) ----
  const int lgrk = J.lgrk, lgrv = J.lgrv;
  float2* tk = reinterpret_cast<float2*>(smem + C::OFF_TK);
  float2* tv = reinterpret_cast<float2*>(smem + C::OFF_TV);
  for (int e = tid; e < (1 << (J.wk + lgrk)); e += nthr) tk[e] = cos_sin_q8(8 * min(e >> lgrk, J.nk - 1), J.nk);
  for (int e = tid; e < (1 << (J.wv + lgrv)); e += nthr) tv[e] = cos_sin_q8(8 * min(e >> lgrv, J.nv - 1), J.nv);
  __syncthreads();

  // ---- this warp's split ----
  const int split = J.split0 + ((int)blockIdx.x - J.cta0) * wpc + warp;
  const int64_t t_begin = (int64_t)(split - J.split0) * kAttSplit;
  if (t_begin >= J.tokens) return;
  const int64_t t_stop = min(J.tokens, t_begin + kAttSplit);
  const int nb = (int)((t_stop - t_begin + kAttBatch - 1) / kAttBatch);
  uint8_t* pb = smem + C::OFF_W + warp * (C::PB + kAttNS * stage);
  uint8_t* stg = pb + C::PB;

  // Stage batch s (tokens t_begin + 32 s ...): six segments in 16-byte
  // chunks, bytes past the last token zero-filled.
  auto issue = [&](int s) {
    if (s < nb) {
      const int64_t row0 = t_begin + (int64_t)s * kAttBatch;
      const int rows = (int)min((int64_t)kAttBatch, J.tokens - row0);
      uint8_t* st = stg + (s % kAttNS) * stage;
      const uint8_t* src[6] = {J.kc + row0 * ak, J.kn + row0 * nbk, J.kh + row0 * 8,
                               J.vc + row0 * av, J.vn + row0 * nbv, J.vh + row0 * 8};
      const int rb[6] = {ak, nbk, hkb, av, nbv, hvb};
      const int off[6] = {0, S_KN, S_KH, S_VA, S_VN, S_VH};
#pragma unroll
      for (int g = 0; g < 6; ++g) {
        const int full = kAttBatch * rb[g], valid = rows * rb[g];
        for (int c = lane * 16; c < full; c += 32 * 16) {
          const int rem = valid - c;
          const int n = rem >= 16 ? 16 : (rem > 0 ? rem : 0);
          cp_async16(st + off[g] + c, n > 0 ? src[g] + c : src[g], n);
        }
      }
    }
    cp_async_commit();
  };

  // ---- lane constants ----
  // K: lane (r, l) takes pairs 8l..8l+7 of token r of each pass of RW tokens;
  // its 8 codes start at bit 8 W l of the row.  A code becomes the byte offset
  // of its table entry (copy lane % 2^lgr) by one rotate and one mask.
  const int r = lane / L, l = lane % L;
  const int wk = J.wk, Tk = 3 + lgrk;
  const int kbit = 8 * wk * l, kwa = kbit >> 5, ksa = kbit & 31;
  const bool kup = ksa + 4 * wk >= 32;                    // codes 4..7 start in the next word
  const int ksb = (ksa + 4 * wk) & 31;
  const uint32_t kC = (uint32_t)(lane & ((1 << lgrk) - 1)) << 3;
  const uint32_t kM = ((1u << wk) - 1u) << Tk;
  int kra[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) kra[j] = (wk * j - Tk) & 31;
  // V: lane owns pairs PV lane .. PV lane + PV - 1; its codes start at bit PV W lane.
  const int wv = J.wv, Tv = 3 + lgrv;
  const int vbit = PV * wv * lane, vwa = vbit >> 5, vsa = vbit & 31;
  const uint32_t vC = (uint32_t)(lane & ((1 << lgrv) - 1)) << 3;
  const uint32_t vM = ((1u << wv) - 1u) << Tv;
  int vra[PV];
#pragma unroll
  for (int j = 0; j < PV; ++j) vra[j] = (wv * j - Tv) & 31;
  const float kinv = J.inv_lk, vinv = J.inv_lv;
  const bool vlog = J.mv == TAC_NORM_LOG;
  const float v2b = J.mv == TAC_NORM_FP32 ? 0.f : (float)(1 << J.bv);

  float m_run[NQ], l_run[NQ];
  float2 acc[NQ][PV];
#pragma unroll
  for (int a = 0; a < NQ; ++a) {
    m_run[a] = -INFINITY;
    l_run[a] = 0.f;
#pragma unroll
    for (int j = 0; j < PV; ++j) acc[a][j] = make_float2(0.f, 0.f);
  }

  // Scores of the batch in `st`: after the passes and the reduction, lane
  // (r, l) holds, for each query, the score of token RW l + r.
  auto scores = [&](const uint8_t* st, float (&keep)[NQ], auto kc_) {
    constexpr int KC = decltype(kc_)::value;
    constexpr bool F32 = KC == 4, LOG = KC == 1 || KC == 3;
    constexpr int KB = KC <= 1 ? 4 : 8;
    // Decoded norms r^ and packed angle codes of this lane's 8 pairs of one token.
    auto load_row = [&](int row, uint32_t& x0, uint32_t& x1, float (&rh)[8]) {
      const uint32_t* arow = reinterpret_cast<const uint32_t*>(st + row * ak);
      const uint32_t w0 = arow[kwa], w1 = arow[kwa + 1], w2 = arow[kwa + 2];
      x0 = __funnelshift_r(w0, w1, ksa);
      x1 = kup ? __funnelshift_r(w1, w2, ksb) : __funnelshift_r(w0, w1, ksb);
      if constexpr (F32) {
        const float4* nr = reinterpret_cast<const float4*>(st + S_KN + row * nbk + 32 * l);
        const float4 n0 = nr[0], n1 = nr[1];
        rh[0] = n0.x; rh[1] = n0.y; rh[2] = n0.z; rh[3] = n0.w;
        rh[4] = n1.x; rh[5] = n1.y; rh[6] = n1.z; rh[7] = n1.w;
      } else {
        const float2 ab = norm_ab(*reinterpret_cast<const float2*>(st + S_KH + row * 8), kinv, (float)(1 << KB), LOG);
        uint32_t nw[2];
        if constexpr (KB == 8) {
          const uint2 v = *reinterpret_cast<const uint2*>(st + S_KN + row * nbk + 8 * l);
          nw[0] = v.x; nw[1] = v.y;
        } else {
          nw[0] = nw[1] = *reinterpret_cast<const uint32_t*>(st + S_KN + row * nbk + 4 * l);
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          constexpr uint32_t NM = ((1u << KB) - 1u) << (23 - KB);
          const int bit = KB * j;
          const uint32_t fb = (rotr(nw[bit >> 5], ((bit & 31) - (23 - KB)) & 31) & NM) | 0x3F800000u;
          float v = __fmaf_rn(__uint_as_float(fb), ab.x, ab.y);
          if constexpr (LOG) v = ex2_approx(v);
          rh[j] = v;
        }
      }
    };
    auto ydec = [&](uint32_t x, int j, float rh) {
      const uint32_t o = (rotr(x, kra[j & 3]) & kM) | kC;
      const float2 c = *reinterpret_cast<const float2*>(reinterpret_cast<const uint8_t*>(tk) + o);
      return mul2(make_float2(rh, rh), c);
    };
    // Partial scores of tokens kA RW + r and kB RW + r over this lane's pairs;
    // each rotated-query granule is loaded once for both.
    auto pass = [&](auto ka_, auto kb_, float (&pa)[NQ], float (&pb)[NQ]) {
      uint32_t xa0, xa1, xb0, xb1;
      float ra[8], rb[8];
      load_row(decltype(ka_)::value * RW + r, xa0, xa1, ra);
      load_row(decltype(kb_)::value * RW + r, xb0, xb1, rb);
      float2 sa[NQ], sb[NQ];
#pragma unroll
      for (int a = 0; a < NQ; ++a) sa[a] = sb[a] = make_float2(0.f, 0.f);
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        const float2 ya0 = ydec(m < 2 ? xa0 : xa1, 2 * m, ra[2 * m]);
        const float2 ya1 = ydec(m < 2 ? xa0 : xa1, 2 * m + 1, ra[2 * m + 1]);
        const float2 yb0 = ydec(m < 2 ? xb0 : xb1, 2 * m, rb[2 * m]);
        const float2 yb1 = ydec(m < 2 ? xb0 : xb1, 2 * m + 1, rb[2 * m + 1]);
#pragma unroll
        for (int a = 0; a < NQ; ++a) {
          const float2* qa = qrot + a * C::QROW + 10 * l + 2 * m;
          const float4 q = NQ >= 4 ? lds_f4_reload(qa) : *reinterpret_cast<const float4*>(qa);
          sa[a] = __ffma2_rn(make_float2(q.x, q.y), ya0, sa[a]);
          sa[a] = __ffma2_rn(make_float2(q.z, q.w), ya1, sa[a]);
          sb[a] = __ffma2_rn(make_float2(q.x, q.y), yb0, sb[a]);
          sb[a] = __ffma2_rn(make_float2(q.z, q.w), yb1, sb[a]);
        }
      }
#pragma unroll
      for (int a = 0; a < NQ; ++a) {
        pa[a] = sa[a].x + sa[a].y;
        pb[a] = sb[a].x + sb[a].y;
      }
    };
    att_tree<L, 0, 1, NQ>(pass, l, keep);
  };

  // V accumulation over the batch's valid tokens: acc += p_t y^V_t.
  auto values = [&](const uint8_t* st, int valid, auto vc_) {
    constexpr int VC = decltype(vc_)::value;
    constexpr bool F32 = VC == 4, LOG = VC == 1 || VC == 3;
    constexpr int VB = VC <= 1 ? 4 : 8;
    constexpr uint32_t NM = ((1u << VB) - 1u) << (23 - VB);
    const int nbit = PV * VB * lane, nwa = nbit >> 5;
    int nra[PV];
#pragma unroll
    for (int j = 0; j < PV; ++j) nra[j] = ((nbit & 31) + VB * j - (23 - VB)) & 31;
#pragma unroll 4
    for (int t = 0; t < valid; ++t) {
      const uint32_t* arow = reinterpret_cast<const uint32_t*>(st + S_VA + t * av);
      const uint32_t x = __funnelshift_r(arow[vwa], arow[vwa + 1], vsa);
      const uint8_t* prow = pb + t * C::PBROW;
      float rh[PV];
      if constexpr (F32) {
        const float* nr = reinterpret_cast<const float*>(st + S_VN + t * nbv) + PV * lane;
        if constexpr (PV == 2) {
          const float2 v = *reinterpret_cast<const float2*>(nr);
          rh[0] = v.x; rh[1] = v.y;
        } else {
          rh[0] = nr[0];
        }
      } else {
        const float2 ab = *reinterpret_cast<const float2*>(prow);
        const uint32_t w = reinterpret_cast<const uint32_t*>(st + S_VN + t * nbv)[nwa];
#pragma unroll
        for (int j = 0; j < PV; ++j) {
          const uint32_t fb = (rotr(w, nra[j]) & NM) | 0x3F800000u;
          float v = __fmaf_rn(__uint_as_float(fb), ab.x, ab.y);
          if constexpr (LOG) v = ex2_approx(v);
          rh[j] = v;
        }
      }
      float2 pp[NQ];
#pragma unroll
      for (int a = 0; a < NQ; a += 2) {
        if (a + 1 < NQ) {
          const float4 q = *reinterpret_cast<const float4*>(prow + 16 + 8 * a);
          pp[a] = make_float2(q.x, q.y);
          pp[a + 1] = make_float2(q.z, q.w);
        } else {
          pp[a] = *reinterpret_cast<const float2*>(prow + 16 + 8 * a);
        }
      }
#pragma unroll
      for (int j = 0; j < PV; ++j) {
        const uint32_t o = (rotr(x, vra[j]) & vM) | vC;
        const float2 cs = *reinterpret_cast<const float2*>(reinterpret_cast<const uint8_t*>(tv) + o);
        const float2 y = mul2(make_float2(rh[j], rh[j]), cs);
#pragma unroll
        for (int a = 0; a < NQ; ++a) acc[a][j] = __ffma2_rn(pp[a], y, acc[a][j]);
      }
    }
  };

  issue(0);
  for (int s = 0; s < nb; ++s) {
    issue(s + 1);
    cp_async_wait<1>();
    __syncwarp();
    const uint8_t* st = stg + (s % kAttNS) * stage;
    const int valid = (int)min((int64_t)kAttBatch, t_stop - (t_begin + (int64_t)s * kAttBatch));

    float keep[NQ];
    switch (J.ck) {
      case 0: scores(st, keep, IC<0>{}); break;
      case 1: scores(st, keep, IC<1>{}); break;
      case 2: scores(st, keep, IC<2>{}); break;
      case 3: scores(st, keep, IC<3>{}); break;
      default: scores(st, keep, IC<4>{}); break;
    }

    // ---- online softmax (base 2); lane (r, l) owns token t = RW l + r ----
    const int t = RW * l + r;
    const bool live = t < valid;
    uint8_t* prow = pb + t * C::PBROW;
    float pw[NQ];
#pragma unroll
    for (int a = 0; a < NQ; ++a) {
      const float sa = live ? keep[a] : -INFINITY;
      float mx = sa;
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      const float mn = fmaxf(m_run[a], mx);
      const float f = ex2_approx(m_run[a] - mn);   // m_run = -inf at first: f = 0
      pw[a] = ex2_approx(sa - mn);
      l_run[a] = __fmaf_rn(l_run[a], f, pw[a]);
      m_run[a] = mn;
#pragma unroll
      for (int j = 0; j < PV; ++j) acc[a][j] = mul2(acc[a][j], make_float2(f, f));
    }
    if (live && J.mv != TAC_NORM_FP32)
      *reinterpret_cast<float2*>(prow) = norm_ab(*reinterpret_cast<const float2*>(st + S_VH + t * 8), vinv, v2b, vlog);
#pragma unroll
    for (int a = 0; a < NQ; a += 2) {
      if (a + 1 < NQ) *reinterpret_cast<float4*>(prow + 16 + 8 * a) = make_float4(pw[a], pw[a], pw[a + 1], pw[a + 1]);
      else *reinterpret_cast<float2*>(prow + 16 + 8 * a) = make_float2(pw[a], pw[a]);
    }
    __syncwarp();

    switch (J.cv) {
      case 0: values(st, valid, IC<0>{}); break;
      case 1: values(st, valid, IC<1>{}); break;
      case 2: values(st, valid, IC<2>{}); break;
      case 3: values(st, valid, IC<3>{}); break;
      default: values(st, valid, IC<4>{}); break;
    }
    __syncwarp();
  }
  cp_async_wait<0>();

  // ---- the split's partial results: (max, sum, accumulator) per query ----
  float* rec = ws + J.ws + (int64_t)(split - J.split0) * nq * att_rec_floats(D);
#pragma unroll
  for (int a = 0; a < NQ; ++a) {
    float ls = l_run[a];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) ls += __shfl_xor_sync(0xffffffffu, ls, o);
    if (a < nq) {
      float* ra = rec + a * att_rec_floats(D);
      if (lane == 0) { ra[0] = m_run[a]; ra[1] = ls; }
#pragma unroll
      for (int j = 0; j < PV; ++j)   // accumulators are per slot; the record holds pairs in order
        *reinterpret_cast<float2*>(ra + 2 + 2 * slot_pair<D>(PV * lane + j)) = acc[a][j];
    }
  }
}

// One CTA of 4 warps per (job, query): warp w merges splits w, w + 4, ...
// against the row's overall max, the warps' sums are added in shared memory,
// and warp 0 normalizes, applies D H (fp32 butterfly) and stores the row.
template <int D, typename TO>
__global__ void __launch_bounds__(128) attend_combine(const __grid_constant__ AttParams p, const float* ws,
                                                      int nrows_total) {
  constexpr int ESZ = (int)sizeof(TO);
  constexpr int E = D / 32;
  __shared__ float part[4][D];
  __shared__ float red[4][2];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = blockIdx.x;                      // global (job, query) index
  if (g >= nrows_total) return;
  int jb = 0, base = 0;
  for (; jb < p.njobs; ++jb) {
    if (g < base + p.job[jb].nq) break;
    base += p.job[jb].nq;
  }
  const AttJob& J = p.job[jb];
  const int a = g - base;
  const int nsp = (int)((J.tokens + kAttSplit - 1) / kAttSplit);
  const float* recs = ws + J.ws + (int64_t)a * att_rec_floats(D);
  const int64_t stride = (int64_t)J.nq * att_rec_floats(D);   // between splits
  float M = -INFINITY;
  for (int s = threadIdx.x; s < nsp; s += 128) M = fmaxf(M, recs[s * stride]);
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  if (lane == 0) red[warp][0] = M;
  __syncthreads();
  M = fmaxf(fmaxf(red[0][0], red[1][0]), fmaxf(red[2][0], red[3][0]));
  float Ls = 0.f;
  float y[E];
#pragma unroll
  for (int e = 0; e < E; ++e) y[e] = 0.f;
#pragma unroll 4
  for (int s = warp; s < nsp; s += 4) {
    const float* ra = recs + s * stride;
    const float f = ex2_approx(ra[0] - M);
    Ls = __fmaf_rn(ra[1], f, Ls);
#pragma unroll
    for (int e = 0; e < E; ++e) y[e] = __fmaf_rn(ra[2 + lane + 32 * e], f, y[e]);
  }
#pragma unroll
  for (int e = 0; e < E; ++e) part[warp][lane + 32 * e] = y[e];
  if (lane == 0) red[warp][1] = Ls;
  __syncthreads();
  if (warp != 0) return;
  const float inv = 1.f / (red[0][1] + red[1][1] + red[2][1] + red[3][1]);
  float* row = part[0];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int j = lane + 32 * e;
    row[j] = (part[0][j] + part[1][j] + part[2][j] + part[3][j]) * inv;
  }
  smem_fwht<D>(row, 1, lane, 32, false);
  const float sc = rsqrtf((float)D);
  uint8_t* orow = reinterpret_cast<uint8_t*>(J.out) + (int64_t)a * J.out_stride * ESZ;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int j = lane + 32 * e;
    float v = row[j] * sc;
    if ((J.sv[j >> 5] >> (j & 31)) & 1u) v = -v;
    if constexpr (ESZ == 2) reinterpret_cast<__nv_bfloat16*>(orow)[j] = __float2bfloat16_rn(v);
    else reinterpret_cast<float*>(orow)[j] = v;
  }
}

// Warps per CTA for a launch: the count (1..kAttMaxWarps) that keeps the most
// warps resident per SM, given the CTA's shared memory (which grows with the
// warps) and the kernel's registers; ties go to more warps per CTA.
static int att_warps_per_cta(int smem_fixed, int smem_per_warp, int regs) {
  constexpr int kSmemSM = 228 * 1024, kSmemCTA = 227 * 1024, kReserved = 1024;
  const int regs_warp = ((regs * 32 + 255) / 256) * 256;
  int best = 1, best_res = -1;
  for (int w = 1; w <= kAttMaxWarps; ++w) {
    const int sm = smem_fixed + w * smem_per_warp;
    if (sm > kSmemCTA) break;
    const int by_smem = kSmemSM / (sm + kReserved);
    const int by_regs = 65536 / (regs_warp * w);
    const int by_warps = 64 / w;
    const int res = std::min(by_smem, std::min(by_regs, by_warps)) * w;
    if (res >= best_res) { best_res = res; best = w; }
  }
  return best;
}

// Launches the partial and combine kernels for one group of jobs.  The CTA
// assignment (cta0 per job, nctas) is made here, after the warps per CTA.
template <int D, typename TQ, int NQ>
static cudaError_t launch_attend_t(const AttParams& p_in, int nrows_total, float* ws, cudaStream_t st) {
  using C = Att<D, NQ>;
  auto kp = attend_partial<D, NQ>;
  // per device, set on the first launch; atomic so that host threads making
  // first calls at once do not race (each sets the same values)
  static std::atomic<int> regs[64];
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (regs[dev].load(std::memory_order_acquire) == 0) {
    cudaError_t e = cudaFuncSetAttribute(kp, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (e != cudaSuccess) return e;
    cudaFuncAttributes fa;
    e = cudaFuncGetAttributes(&fa, kp);
    if (e != cudaSuccess) return e;
    regs[dev].store(fa.numRegs > 0 ? fa.numRegs : 1, std::memory_order_release);
  }
  AttParams p = p_in;
  int stage = 0;
  for (int j = 0; j < p.njobs; ++j) {
    const AttJob& J = p.job[j];
    stage = std::max(stage, att_stage_bytes(D, J.wk, J.bk, J.mk, J.wv, J.bv, J.mv));
  }
  const int wpc = att_warps_per_cta(C::smem(stage, 0), C::smem(stage, 1) - C::smem(stage, 0), regs[dev].load(std::memory_order_relaxed));
  int64_t ctas = 0;
  for (int j = 0; j < p.njobs; ++j) {
    AttJob& J = p.job[j];
    const int64_t ns = (J.tokens + kAttSplit - 1) / kAttSplit;
    J.cta0 = (int32_t)ctas;
    ctas += (ns + wpc - 1) / wpc;
  }
  p.nctas = (int32_t)ctas;
  if (p.nctas > 0) kp<<<p.nctas, 32 * wpc, C::smem(stage, wpc), st>>>(p, ws);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (nrows_total > 0) attend_combine<D, TQ><<<nrows_total, 128, 0, st>>>(p, ws, nrows_total);
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
