// Internal definitions shared by the libtac CUDA translation units (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/tac.h"

namespace tac {

constexpr int kMinBlocks = 2;      // resident CTAs per SM the encode / decode kernels are built for
constexpr int kPairsPerThread = 8; // each thread owns 8 consecutive angle pairs (16 elements)
constexpr int kMaxW = 8;           // code bits <= 8 (n <= 256)
// Tables holding one entry per bin for every supported n back to back:
// n = 2, 4, ..., 256 (510 entries), then n = 48 and n = 56 (Table 1).
constexpr int kTabEntries = 616;
constexpr float kU = 5.9604644775390625e-08f;  // fp32 unit roundoff 2^-24

// Lookup tables indexed by a per-pair code are replicated: entry e of copy c
// sits at index e*R + c and lane l reads copy l % R, so the 16 lanes a 64-bit
// shared load serves at a time spread over 16 bank pairs (conflict-free for
// R = 16; for smaller R two or four lanes share a bank pair).  R is the largest
// power of two <= 16 with n * R * 8 <= the byte budget.
__host__ __device__ constexpr int tab_copies(int n, int budget) {
  int r = 16;
  while (r > 1 && n * r * 8 > budget) r >>= 1;
  return r;
}

__host__ __device__ constexpr bool is_pow2(int n) { return n > 0 && (n & (n - 1)) == 0; }
// Code bits for n bins: ceil(log2 n).
__host__ __device__ constexpr int code_bits(int n) {
  int w = 0;
  while ((1 << w) < n) ++w;
  return w;
}
// Offset of the table for n bins inside the table of every supported n.
__host__ __device__ constexpr int tab_offset_n(int n) { return is_pow2(n) ? n - 2 : (n == 48 ? 510 : 558); }
// The n of table entry idx and the entry's index within that n's table.
__host__ __device__ constexpr int tab_n_of(int idx) {
  if (idx >= 558) return 56;
  if (idx >= 510) return 48;
  int w = 1;
  while ((1 << (w + 1)) - 2 <= idx) ++w;
  return 1 << w;
}

// ---------------------------------------------------------------------------
// Geometry for head dimension D.  P = D/2 angle pairs per row; each lane owns 8
// pairs, so L = P/8 lanes share a row and a warp covers RW = 32/L rows (its
// "warp tile").  Every warp runs its own pipeline over warp tiles.
// ---------------------------------------------------------------------------
template <int D>
struct Geo {
  static constexpr int P = D / 2;
  static constexpr int L = P / kPairsPerThread;
  static constexpr int RW = 32 / L;
  static constexpr int LOGD = (D == 16) ? 4 : (D == 32) ? 5 : (D == 64) ? 6 : 7;
  // Transpose buffer (L > 1): pair i of warp-tile row r at r*ST + the offset
  // of i in its pair row, (i / L)*SM + 8*((i % L) ^ s), where for L = 4 the two
  // 16-byte granules of pair rows 4..7 trade places (s = 2 there, else 0).
  // Two patterns use it: lane l touches pairs l + L*m (m = 0..7, 8-byte
  // accesses at m*SM + 8*(l ^ swa(m))) and pairs 8l..8l+7 as four 16-byte
  // granules (at (8/L)*l*SM + tp_pair(2q ^ swb(l))).  SM, ST and the swap make
  // both patterns free of bank conflicts (a shared-memory model of 16-lane
  // phases for 8-byte and 8-lane phases for 16-byte accesses: 16 wavefronts
  // each per warp tile); for L = 4 no padding alone does (one of the two then
  // takes 32).
  static constexpr int SM = L == 8 ? 80 : L == 4 ? 32 : 16;
  static constexpr int ST = L == 8 ? 704 : L == 4 ? 288 : 144;
  static constexpr int TP_W = (L > 1) ? RW * ST : 0;
  __host__ __device__ static constexpr int swa(int m) { return L == 4 ? ((m >> 1) & 2) : 0; }
  __host__ __device__ static constexpr int swb(int l) { return L == 4 ? (l & 2) : 0; }
  __host__ __device__ static constexpr int tp_pair(int i) { return (i / L) * SM + (i % L) * 8; }
};

// Row-major element rows of a warp tile with a per-row pad such that lane l of a
// row reading pair l + L*m (bytes [2i*ESZ, 2i*ESZ + 2*ESZ)) hits distinct banks
// across the rows of the warp; rows start on 16-byte boundaries.
template <int D, int ESZ>
struct RowTile {
  static constexpr int ROWB = D * ESZ;
  static constexpr int CPR = ROWB / 16;
  static constexpr int SPAN = 2 * ESZ * Geo<D>::L;
  // padded row pitch: the 16-byte run loads of two bf16 rows of d = 64 (one
  // quarter-warp) fall on disjoint banks when the pitch is 64 mod 128
  static constexpr int STRIDE = ROWB + ((D == 64 && ESZ == 2) ? 64 : (SPAN > 16 ? SPAN : 16));
  static constexpr int BYTES = Geo<D>::RW * STRIDE;            // one warp tile
  static constexpr int CHUNKS = Geo<D>::RW * CPR / 32;         // 16-byte chunks per lane
};

// Record order (reading R9): slot v of a record holds the code of pair
// phi_d(v).  For d = 64 and 128 (L = d/16), phi(v) = 4 (v mod L) + ((v / L)
// mod 4) + 4 L floor(v / 4L): the kernels work in slot order throughout, and
// the slots l + L m (m = 0..7) a lane loads (encode) or stores (decode) are the
// pairs 4 l + (m mod 4) + 4 L (m / 4), two runs of 4 consecutive pairs.  For
// d <= 32 the order is natural.
template <int D>
__host__ __device__ constexpr bool run_layout() { return D == 64 || D == 128; }
template <int D>
__host__ __device__ constexpr int slot_pair(int v) {
  if constexpr (run_layout<D>()) {
    constexpr int L = D / 16;
    return 4 * (v % L) + (v / L) % 4 + 4 * L * (v / (4 * L));
  } else {
    return v;
  }
}

// The slot that holds pair i (the inverse of slot_pair).
template <int D>
__host__ __device__ constexpr int pair_slot(int i) {
  if constexpr (run_layout<D>()) {
    constexpr int L = D / 16;
    return (i / 4) % L + L * ((i % 4) + 4 * (i / (4 * L)));
  } else {
    return i;
  }
}

// ---------------------------------------------------------------------------
// Device job descriptors (kernel parameters, copied by value at launch).
// ---------------------------------------------------------------------------
struct EncJob {
  const void* x;       // input rows
  uint8_t* codes;      // angle plane base
  uint8_t* norms;      // norm plane base
  uint8_t* hdr;        // header plane base (float2 per slot)
  const int64_t* slot; // destination slots or nullptr
  uint32_t* status;    // gets TAC_E_NONFINITE when a row holds a NaN or an inf (or nullptr)
  int64_t capacity;    // record slots of the destination planes
  int64_t rows;
  int64_t stride;      // elements
  uint32_t signs[4];
  int32_t w;           // log2 n
  int32_t b;           // norm bits (4 or 8)
  int32_t mode;        // 0 linear, 1 log
  int32_t tile0;       // first global tile of this job
};

static_assert(sizeof(EncJob) == 104 && sizeof(EncJob) % 8 == 0, "EncJob: the workspace copy is sized by it");

struct EncParams {
  int32_t njobs;
  int32_t ntiles;
  // Re-decision queue of the launch (workspace, see the encode kernel): the
  // codes the fast path could not certify, 32-byte entries.
  uint4* gq;                   // gq_cap entries (two uint4 each)
  unsigned long long* gq_n;    // entries appended (may pass gq_cap: the rest went to ovf)
  uint32_t* ovf;               // one bit per warp-tile row (tile * RW + row in tile): rows
                               // whose entries found the queue full, re-decided whole
  int64_t gq_cap;
  EncJob* gjobs;               // workspace copy of job[0, njobs), written by the encode kernel
  EncJob job[TAC_MAX_JOBS];
};

// Parameters of the encode's fix-up kernel (small: the job table is read from
// the copy the encode kernel leaves in the workspace).
struct FixParams {
  const EncJob* job;
  uint4* gq;
  unsigned long long* gq_n;
  uint32_t* ovf;
  int64_t gq_cap;
  int32_t njobs;
  int32_t ntiles;
};

struct DecJob {
  const uint8_t* codes;
  const uint8_t* norms;
  const uint8_t* hdr;
  const int64_t* slot;
  int64_t capacity;
  void* y;
  int64_t rows;
  int64_t stride;      // elements
  uint32_t signs[4];
  int32_t w;
  int32_t b;
  int32_t mode;
  int32_t tile0;
};

struct DecParams {
  int32_t njobs;
  int32_t ntiles;
  DecJob job[TAC_MAX_JOBS];
};

// Job owning global tile t (jobs are sorted by tile0, job 0 starts at tile 0).
template <typename Params>
__device__ __forceinline__ int find_job(const Params& p, int t) {
  int lo = 0, hi = p.njobs - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (p.job[mid].tile0 <= t) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// XOR masks flipping the IEEE sign bits of elements 2i and 2i+1 where s_j = -1
// (D of Sec. 2).  bf16 pairs share one 32-bit word (bits 15 and 31); fp32 pairs
// use one word each.
template <int ESZ>
__device__ __forceinline__ uint2 pair_sign_mask(const uint32_t* signs, int i) {
  const uint32_t two = (signs[(2 * i) >> 5] >> ((2 * i) & 31)) & 3u;
  if constexpr (ESZ == 2) return make_uint2(((two & 1u) << 15) | ((two >> 1) << 31), 0u);
  else return make_uint2((two & 1u) << 31, (two >> 1) << 31);
}

// ---------------------------------------------------------------------------
// Exact-symmetry trig tables.  Every table entry is (cos, sin) of 2 pi Q / (8 n)
// for an integer Q: the angle is reduced to an octant with integer arithmetic
// and evaluated with sincospif on [0, pi/4], so entries that are equal or
// negated by symmetry are bit-identical (needed for the exact tie behaviour of
// the edge test at multiples of pi/4).
// ---------------------------------------------------------------------------
__device__ __forceinline__ float2 cos_sin_q8(int Q, int n) {
  const int N8 = 8 * n;
  Q %= N8;
  if (Q < 0) Q += N8;
  const int o = Q / n;       // octant 0..7
  const int rem = Q - o * n; // 0..n-1
  float c, s;
  int quarter;
  if ((o & 1) == 0) {        // angle = (o/2) pi/2 + beta, beta = pi rem / (4n)
    quarter = o >> 1;
    if (rem == 0) { s = 0.f; c = 1.f; }
    else sincospif((float)rem / (float)(4 * n), &s, &c);
  } else {                   // angle = ((o+1)/2) pi/2 - beta', beta' = pi (n - rem)/(4n)
    quarter = (o + 1) >> 1;
    const int rr = n - rem;  // 1..n; rr == n is beta' = pi/4 exactly
    if (rr == n) { s = 0.70710678118654752f; c = 0.70710678118654752f; }
    else sincospif((float)rr / (float)(4 * n), &s, &c);
    s = -s;                  // (cos(-b'), sin(-b'))
  }
  switch (quarter & 3) {     // rotate (c, s) by quarter * pi/2
    case 0: return make_float2(c, s);
    case 1: return make_float2(-s, c);
    case 2: return make_float2(-c, -s);
    default: return make_float2(s, -c);
  }
}

// ---------------------------------------------------------------------------
// Edge directions for the exact-decision path, built by the host compiler in
// fp64: cos/sin from their Taylor series on [0, pi/4] (|x| <= 0.79: 24 terms
// reach full double precision) with the same integer octant reduction as above.
// ---------------------------------------------------------------------------
namespace cx {
struct CS { double c, s; };
constexpr double kPi = 3.141592653589793238462643383279502884;
constexpr double sin_series(double x) {
  double term = x, sum = x;
  for (int k = 1; k < 24; ++k) { term *= -x * x / ((2.0 * k) * (2.0 * k + 1.0)); sum += term; }
  return sum;
}
constexpr double cos_series(double x) {
  double term = 1.0, sum = 1.0;
  for (int k = 1; k < 24; ++k) { term *= -x * x / ((2.0 * k - 1.0) * (2.0 * k)); sum += term; }
  return sum;
}
constexpr CS cos_sin_q8(int Q, int n) {
  const int N8 = 8 * n;
  Q %= N8;
  if (Q < 0) Q += N8;
  const int o = Q / n, rem = Q - o * n;
  double c = 1.0, s = 0.0;
  int quarter = 0;
  if ((o & 1) == 0) {
    quarter = o >> 1;
    if (rem != 0) { const double a = kPi * rem / (4.0 * n); c = cos_series(a); s = sin_series(a); }
  } else {
    quarter = (o + 1) >> 1;
    const int rr = n - rem;
    if (rr == n) { c = 0.70710678118654752440; s = 0.70710678118654752440; }
    else { const double a = kPi * rr / (4.0 * n); c = cos_series(a); s = sin_series(a); }
    s = -s;
  }
  switch (quarter & 3) {
    case 0: return CS{c, s};
    case 1: return CS{-s, c};
    case 2: return CS{-c, -s};
    default: return CS{s, -c};
  }
}
}  // namespace cx

// Encode edge table for n bins, entry e: direction psi_e = phi_e + pi/4 of the
// edge phi_e = (e + 1/2) 2 pi / n between bins e and e+1, as (cos psi, sin psi).
// In the pair's butterfly halves (E, O) = ((y0 + y1)/2, (y0 - y1)/2) the sign of
// E cos psi - O sin psi equals the sign of sin(theta - phi_e) (Alg. 1 angle).
__device__ __forceinline__ int edge_q8(int e, int n) { return 8 * e + 4 + n; }

// Decode table for n bins, entry k: (cos phi_k + sin phi_k, cos phi_k - sin phi_k)
// = sqrt2 (sin(phi_k + pi/4), cos(phi_k + pi/4)), phi_k = 2 pi k / n (Sec. 3.1).
__device__ __forceinline__ int centre_q8(int k, int n) { return 8 * k + n; }

// ---------------------------------------------------------------------------
// cp.async (sm_80+ async global -> shared copies, 16 bytes, zero-fill tail).
// ---------------------------------------------------------------------------
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, int src_bytes) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

// ---------------------------------------------------------------------------
// Packed fp32 pairs (sm_100 FADD2/FFMA2).  a - b is formed as fma(b, -1, a),
// which rounds exactly like a - b.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float2 add2(float2 a, float2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {
  return __ffma2_rn(b, make_float2(-1.f, -1.f), a);
}
__device__ __forceinline__ float2 mul2(float2 a, float2 b) { return __fmul2_rn(a, b); }

// In-register butterfly over the 8 values of v: the stages on index bits with
// HLO <= 2^bit < HHI (<1, 8>: all three).
template <int HHI = 8, int HLO = 1>
__device__ __forceinline__ void butterfly8(float2 (&v)[8]) {
#pragma unroll
  for (int h = HLO; h < HHI; h <<= 1) {
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      if ((m & h) == 0) {
        const float2 a = v[m], b = v[m + h];
        v[m] = add2(a, b);
        v[m + h] = sub2(a, b);
      }
    }
  }
}

// bf16 <-> fp32 (exact widening; bf16 is the high half of an fp32).
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// Hardware approximations (MUFU): relative error of a few fp32 ulp.
__device__ __forceinline__ float sqrt_approx(float x) {
  float r; asm("sqrt.approx.f32 %0, %1;" : "=f"(r) : "f"(x)); return r;
}
__device__ __forceinline__ float rcp_approx(float x) {
  float r; asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x)); return r;
}
__device__ __forceinline__ float lg2_approx(float x) {
  float r; asm("lg2.approx.f32 %0, %1;" : "=f"(r) : "f"(x)); return r;
}
__device__ __forceinline__ float ex2_approx(float x) {
  float r; asm("ex2.approx.f32 %0, %1;" : "=f"(r) : "f"(x)); return r;
}
// Flush-to-zero forms (subnormal inputs and results read as zero): the callers
// keep their arguments and results in the normal range.
__device__ __forceinline__ float sqrt_ftz(float x) {
  float r; asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x)); return r;
}
__device__ __forceinline__ float lg2_ftz(float x) {
  float r; asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x)); return r;
}
__device__ __forceinline__ float ex2_ftz(float x) {
  float r; asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x)); return r;
}
__device__ __forceinline__ float min3(float a, float b, float c) {
  float r; asm("min.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c)); return r;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
  float r; asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c)); return r;
}

}  // namespace tac
