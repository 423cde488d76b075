// Attention jobs and launch parameters shared by the C ABI (tac_api.cu) and
// the attention kernels (tac_attend.cu).
#pragma once
#include "tac_common.cuh"

namespace tac {

// Attention jobs (tac_attend_multi): record planes, runtime codebooks, queries.
struct AttJob {
  const uint8_t* kc; const uint8_t* kn; const uint8_t* kh;   // K planes (angle, norm, header)
  const uint8_t* vc; const uint8_t* vn; const uint8_t* vh;   // V planes
  const void* q; void* out;
  int64_t q_stride, out_stride;      // elements
  int64_t tokens;
  float scale;
  int32_t nq;
  int32_t nk, wk, bk, mk;            // K: bins, code bits, norm bits, norm mode
  int32_t nv, wv, bv, mv;            // V
  float inv_lk, inv_lv;              // 1 / (2^b - 1) of K and V norms (0 for fp32 norms)
  int32_t lgrk, lgrv;                // log2 of the bin-centre table copies (K, V)
  int32_t ck, cv;                    // norm case (att_norm_case) of K and V
  uint32_t sk[4], sv[4];             // D of K and of V
  int32_t split0;                    // first global split of this job
  int32_t cta0;                      // first CTA of this job
  int64_t ws;                        // first workspace float of this job
};

struct AttParams {
  int32_t njobs;
  int32_t nctas;
  int32_t nsplits;
  int32_t q_bf16;                    // queries (and outputs) are bf16 rows, else fp32
  AttJob job[TAC_ATTEND_MAX_JOBS];   // 200 bytes each: within the 32 KB of kernel parameters
};

// Per-split workspace record: max (log2 units), sum, accumulator (d floats).
__host__ __device__ constexpr int att_rec_floats(int d) { return d + 2; }

// Attention staging: a warp takes its split in batches of 32 tokens; one
// staged batch holds 32 rows of each record plane (K angle | K norm | K header |
// V angle | V norm | V header, headers absent for fp32 norms) plus 16 bytes of
// slack for word reads past a row's end.
constexpr int kAttBatch = 32;
constexpr int kAttTabBytes = 4096;   // per bin-centre table, all copies
__host__ __device__ inline int att_stage_bytes(int d, int wk, int bk, int mk, int wv, int bv, int mv) {
  const int P = d / 2;
  return kAttBatch * (P * wk / 8 + P * bk / 8 + (mk != TAC_NORM_FP32 ? 8 : 0) + P * wv / 8 + P * bv / 8 +
                      (mv != TAC_NORM_FP32 ? 8 : 0)) +
         16;
}
// Norm decoding case: 0/1 = 4-bit linear/log, 2/3 = 8-bit linear/log, 4 = fp32.
__host__ __device__ inline int att_norm_case(int bits, int mode) {
  return mode == TAC_NORM_FP32 ? 4 : (bits == 8 ? 2 : 0) + (mode == TAC_NORM_LOG ? 1 : 0);
}
// log2 of the copies of an n-entry (cos, sin) table within kAttTabBytes (<= 16).
__host__ __device__ inline int att_table_lgr(int n) {
  int lg = 0;
  while (lg < 4 && (n << (lg + 1)) * 8 <= kAttTabBytes) ++lg;
  return lg;
}

}  // namespace tac
