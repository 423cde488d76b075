// Internal definitions shared by the libtac CUDA translation units (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/tac.h"

namespace tac {

constexpr int kTileRows = 128;     // rows per tile: one thread per row
constexpr int kThreads = 128;      // threads per CTA
constexpr int kMaxW = 8;           // log2 n <= 8 (n <= 256)
constexpr int kTabEntries = 512;   // sum_{w=1..8} 2^w = 510, padded
constexpr float kU = 5.9604644775390625e-08f;  // fp32 unit roundoff 2^-24

// Offset of the table for n = 2^w inside a table holding every w = 1..8 back to back.
__host__ __device__ constexpr int tab_offset(int w) { return (1 << w) - 2; }

// ---------------------------------------------------------------------------
// Device job descriptors (kernel parameters, copied by value at launch).
// ---------------------------------------------------------------------------
struct EncJob {
  const void* x;       // input rows
  uint8_t* codes;      // angle plane base
  uint8_t* norms;      // norm plane base
  uint8_t* hdr;        // header plane base (float2 per slot)
  const int64_t* slot; // destination slots or nullptr
  int64_t capacity;    // record slots of the destination planes
  int64_t rows;
  int64_t stride;      // elements
  uint32_t signs[4];
  int32_t w;           // log2 n
  int32_t b;           // norm bits (4 or 8)
  int32_t mode;        // 0 linear, 1 log
  int32_t tile0;       // first global tile of this job
};

struct EncParams {
  int32_t njobs;
  int32_t ntiles;
  EncJob job[TAC_MAX_JOBS];
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
  // rotate (c, s) by quarter * pi/2
  switch (quarter & 3) {
    case 0: return make_float2(c, s);
    case 1: return make_float2(-s, c);
    case 2: return make_float2(-c, -s);
    default: return make_float2(s, -c);
  }
}

// Same construction in fp64 for the exact-decision path.
__device__ __forceinline__ double2 cos_sin_q8_d(int Q, int n) {
  const int N8 = 8 * n;
  Q %= N8;
  if (Q < 0) Q += N8;
  const int o = Q / n;
  const int rem = Q - o * n;
  double c, s;
  int quarter;
  if ((o & 1) == 0) {
    quarter = o >> 1;
    if (rem == 0) { s = 0.0; c = 1.0; }
    else sincospi((double)rem / (double)(4 * n), &s, &c);
  } else {
    quarter = (o + 1) >> 1;
    const int rr = n - rem;
    if (rr == n) { s = 0.70710678118654752440; c = 0.70710678118654752440; }
    else sincospi((double)rr / (double)(4 * n), &s, &c);
    s = -s;
  }
  switch (quarter & 3) {
    case 0: return make_double2(c, s);
    case 1: return make_double2(-s, c);
    case 2: return make_double2(-c, -s);
    default: return make_double2(s, -c);
  }
}

// Encode edge table for n = 2^w, entry e: direction psi_e = phi_e + pi/4 of the
// edge phi_e = (e + 1/2) 2 pi / n between bins e and e+1, as (cos psi, sin psi).
// In the pair's butterfly halves (E, O) = ((y0 + y1)/2, (y0 - y1)/2) the sign of
// E cos psi - O sin psi equals the sign of sin(theta - phi_e) (Alg. 1 angle).
__device__ __forceinline__ int edge_q8(int e, int n) { return 8 * e + 4 + n; }

// Decode table for n = 2^w, entry k: (cos phi_k + sin phi_k, cos phi_k - sin phi_k)
// = sqrt2 (sin(phi_k + pi/4), cos(phi_k + pi/4)), phi_k = 2 pi k / n (Sec. 3.1).
__device__ __forceinline__ int centre_q8(int k, int n) { return 8 * k + n; }

// ---------------------------------------------------------------------------
// Shared-memory tile swizzle: the 16-byte chunk c of tile row r is stored at
// chunk c ^ sw(r) of that row, so that one thread per row reading chunk c hits
// eight distinct 16-byte bank groups per eight consecutive rows.
// ---------------------------------------------------------------------------
template <int ROWB>
__device__ __forceinline__ int row_swz(int r) {
  constexpr int CPR = ROWB / 16;
  if constexpr (ROWB >= 128) return r & 7;
  else if constexpr (ROWB == 64) return (r >> 1) & (CPR - 1);
  else if constexpr (ROWB == 32) return (r >> 2) & (CPR - 1);
  else return 0;
}

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

// bf16 <-> fp32 (exact widening; bf16 is the high half of an fp32).
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

}  // namespace tac
