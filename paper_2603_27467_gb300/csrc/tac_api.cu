// libtac C ABI: argument checking, plane geometry, rate accounting, the sign
// generator and the batched launch planner.  Kernels live in tac_encode.cu,
// tac_decode.cu and tac_fwht_debug.cu.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "tac_attend.cuh"

namespace tac {
cudaError_t launch_encode_16_bf16(const EncParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st, int phase);
cudaError_t launch_encode_32_bf16(const EncParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st, int phase);
cudaError_t launch_encode_64_bf16(const EncParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st, int phase);
cudaError_t launch_encode_128_bf16(const EncParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st, int phase);
cudaError_t launch_encode_16_f32(const EncParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st, int phase);
cudaError_t launch_encode_32_f32(const EncParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st, int phase);
cudaError_t launch_encode_64_f32(const EncParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st, int phase);
cudaError_t launch_encode_128_f32(const EncParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st, int phase);
cudaError_t launch_decode_16_bf16(const DecParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st);
cudaError_t launch_decode_32_bf16(const DecParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st);
cudaError_t launch_decode_64_bf16(const DecParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st);
cudaError_t launch_decode_128_bf16(const DecParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st);
cudaError_t launch_decode_16_f32(const DecParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st);
cudaError_t launch_decode_32_f32(const DecParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st);
cudaError_t launch_decode_64_f32(const DecParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st);
cudaError_t launch_decode_128_f32(const DecParams& p, int n, int b, int mode, int sms,
                                 cudaStream_t st);

// phase: 1 the encode kernel, 2 its fix-up, 3 both in order (one stream).
static cudaError_t launch_encode(int d, int dtype, int n, int b, int mode, const EncParams& p, int sms,
                                 cudaStream_t st, int phase) {
  const bool bf = dtype == TAC_BF16;
  switch (d) {
    case 16: return bf ? launch_encode_16_bf16(p, n, b, mode, sms, st, phase) : launch_encode_16_f32(p, n, b, mode, sms, st, phase);
    case 32: return bf ? launch_encode_32_bf16(p, n, b, mode, sms, st, phase) : launch_encode_32_f32(p, n, b, mode, sms, st, phase);
    case 64: return bf ? launch_encode_64_bf16(p, n, b, mode, sms, st, phase) : launch_encode_64_f32(p, n, b, mode, sms, st, phase);
    case 128: return bf ? launch_encode_128_bf16(p, n, b, mode, sms, st, phase) : launch_encode_128_f32(p, n, b, mode, sms, st, phase);
  }
  return cudaErrorInvalidValue;
}

static cudaError_t launch_decode(int d, int dtype, int n, int b, int mode, const DecParams& p, int sms,
                                 cudaStream_t st) {
  const bool bf = dtype == TAC_BF16;
  switch (d) {
    case 16: return bf ? launch_decode_16_bf16(p, n, b, mode, sms, st) : launch_decode_16_f32(p, n, b, mode, sms, st);
    case 32: return bf ? launch_decode_32_bf16(p, n, b, mode, sms, st) : launch_decode_32_f32(p, n, b, mode, sms, st);
    case 64: return bf ? launch_decode_64_bf16(p, n, b, mode, sms, st) : launch_decode_64_f32(p, n, b, mode, sms, st);
    case 128: return bf ? launch_decode_128_bf16(p, n, b, mode, sms, st) : launch_decode_128_f32(p, n, b, mode, sms, st);
  }
  return cudaErrorInvalidValue;
}
cudaError_t launch_attend(int d, int dtype, int nq_max, const AttParams& p, int nrows_total, float* ws,
                          cudaStream_t st);
cudaError_t attend_static_workspace(float** ws);
cudaError_t launch_fwht_debug(int d, const void* x, int dtype, int64_t rows, int64_t stride,
                              const uint32_t* signs, float* y, cudaStream_t st);
cudaError_t launch_hw_approx(int op, const float* x, float* y, int64_t n, int sms, cudaStream_t st);
}  // namespace tac

namespace {

thread_local std::string g_err;

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}

int ok() {
  g_err.clear();
  return TAC_OK;
}

int log2_exact(int v) {
  if (v <= 0 || (v & (v - 1))) return -1;
  int w = 0;
  while ((1 << w) < v) ++w;
  return w;
}

// SplitMix64 (Steele, Lea, Flood 2014): output #i of the stream seeded with z.
uint64_t splitmix64(uint64_t z, uint64_t i) {
  z += (i + 1u) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

int check_cfg(const tac_layer_cfg* c, const char* who) {
  if (!c) return fail(TAC_E_INVAL, "%s: cfg is NULL", who);
  if (c->d != 16 && c->d != 32 && c->d != 64 && c->d != 128) {
    if (c->d > 0 && log2_exact(c->d) >= 1)
      return fail(TAC_E_UNSUPPORTED, "%s: d = %d not implemented (16, 32, 64, 128)", who, c->d);
    return fail(TAC_E_INVAL, "%s: d = %d is not a power of two", who, c->d);
  }
  const int n = c->n_angle;
  if (n < 2) return fail(TAC_E_INVAL, "%s: n = %d", who, n);
  const int w = log2_exact(n);
  if (w < 0 && n != 48 && n != 56)
    return fail(TAC_E_UNSUPPORTED, "%s: n = %d not implemented (powers of two 2..256, 48, 56)", who, n);
  if (w > 8) return fail(TAC_E_UNSUPPORTED, "%s: n = %d outside 2..256", who, n);
  if (c->norm_mode != TAC_NORM_LINEAR && c->norm_mode != TAC_NORM_LOG && c->norm_mode != TAC_NORM_FP32)
    return fail(TAC_E_INVAL, "%s: norm_mode = %d", who, c->norm_mode);
  if (c->norm_mode == TAC_NORM_FP32) {
    if (c->norm_bits != 32) return fail(TAC_E_INVAL, "%s: norm_bits = %d with fp32 norms (must be 32)", who, c->norm_bits);
  } else if (c->norm_bits != 4 && c->norm_bits != 8) {
    if (c->norm_bits >= 1 && c->norm_bits <= 16)
      return fail(TAC_E_UNSUPPORTED, "%s: norm_bits = %d not implemented (4, 8)", who, c->norm_bits);
    return fail(TAC_E_INVAL, "%s: norm_bits = %d", who, c->norm_bits);
  }
  return TAC_OK;
}

int64_t angle_row_bytes(const tac_layer_cfg* c) { return (int64_t)(c->d / 2) * tac::code_bits(c->n_angle) / 8; }
int64_t norm_row_bytes(const tac_layer_cfg* c) { return (int64_t)(c->d / 2) * c->norm_bits / 8; }
int64_t header_offset(const tac_layer_cfg* c, int64_t cap) { return (cap * norm_row_bytes(c) + 15) & ~(int64_t)15; }

// Rows per warp tile: 32 lanes, d/16 lanes per row (8 angle pairs per lane).
int64_t tile_rows(int d) { return (int64_t)32 / (d / 16); }

int esize(int dtype) { return dtype == TAC_BF16 ? 2 : dtype == TAC_FP32 ? 4 : 0; }

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

int check_rows(const tac_rows* r, int d, const char* who, const char* name, bool rows16 = true) {
  if (!r) return fail(TAC_E_INVAL, "%s: %s is NULL", who, name);
  if (!esize(r->dtype)) return fail(TAC_E_INVAL, "%s: %s.dtype = %d", who, name, r->dtype);
  if (r->rows < 0) return fail(TAC_E_INVAL, "%s: %s.rows = %lld", who, name, (long long)r->rows);
  if (r->rows == 0) return TAC_OK;
  if (!r->data) return fail(TAC_E_INVAL, "%s: %s.data is NULL", who, name);
  if (!aligned16(r->data)) return fail(TAC_E_INVAL, "%s: %s.data is not 16-byte aligned", who, name);
  if (r->row_stride < d) return fail(TAC_E_INVAL, "%s: %s.row_stride %lld < d %d", who, name, (long long)r->row_stride, d);
  if (rows16 && (r->row_stride * esize(r->dtype)) % 16)
    return fail(TAC_E_INVAL, "%s: %s.row_stride * sizeof(element) is not a multiple of 16", who, name);
  if (r->rows > ((int64_t)1 << 38)) return fail(TAC_E_UNSUPPORTED, "%s: %s.rows too large", who, name);
  return TAC_OK;
}

// SMs each launch of a multi-launch call may use.  A large call gives every
// launch the whole GPU: they run back to back in effect, each at full rate.  A
// small one (fewer than kSplitTiles warp tiles per SM in all) is dominated by
// each launch's ramp (table set-up, first prefetches) and tail, so its launches
// get shares of the SMs in proportion to their tiles (at least one each) and
// run side by side, paying the ramp once.
constexpr int64_t kSplitTiles = 640;   // 32 tiles per warp at 20 warps per SM
void sm_shares(const int64_t* tiles, int ngroups, int sms, int* caps) {
  int64_t total = 0;
  for (int g = 0; g < ngroups; ++g) total += tiles[g];
  if (ngroups <= 1 || total >= kSplitTiles * sms) {
    for (int g = 0; g < ngroups; ++g) caps[g] = sms;
    return;
  }
  int used = 0;
  for (int g = 0; g < ngroups; ++g) {
    caps[g] = (int)std::max<int64_t>(1, tiles[g] * sms / total);
    used += caps[g];
  }
  // hand the SMs left by rounding down to the largest groups (groups are
  // sorted largest first); more groups than SMs may oversubscribe: the extra
  // CTAs wait for a free slot
  for (int g = 0; used < sms && ngroups > 0; g = (g + 1) % ngroups, ++used) ++caps[g];
}

int num_sms() {
  static std::atomic<int> cache[64];   // per device; concurrent first calls store the same value
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (dev < 0 || dev >= 64) return 0;
  int v = cache[dev].load(std::memory_order_relaxed);
  if (!v) {
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    cache[dev].store(v, std::memory_order_relaxed);
  }
  return v;
}

void copy_signs(uint32_t* dst, const tac_layer_cfg* c) {
  for (int q = 0; q < 4; ++q) dst[q] = c->signs[q];
  // bits beyond d are never read by the kernels; clear them for determinism
  if (c->d < 128) {
    for (int q = 0; q < 4; ++q) {
      const int lo = 32 * q;
      if (lo >= c->d) dst[q] = 0u;
      else if (c->d - lo < 32) dst[q] &= (1u << (c->d - lo)) - 1u;
    }
  }
}

}  // namespace

extern "C" {

const char* tac_last_error(void) { return g_err.c_str(); }

const char* tac_version(void) { return "libtac 0.1.0 (TurboAngle encode/decode, sm_103a)"; }

}  // extern "C"

namespace {
// Sign words of the stream keyed by output #q of the SplitMix64 stream seeded with seed.
int make_signs_q(const char* who, uint64_t seed, uint64_t q, int d, uint32_t* out_words) {
  if (!out_words) return fail(TAC_E_INVAL, "%s: out_words is NULL", who);
  if (d < 1 || d > (1 << 20)) return fail(TAC_E_INVAL, "%s: d = %d", who, d);
  const uint64_t key = splitmix64(seed, q);
  const int nw = (d + 31) / 32;
  for (int i = 0; i < nw; ++i) out_words[i] = 0u;
  for (int j = 0; j < d; ++j)
    if (splitmix64(key, (uint64_t)j) >> 63) out_words[j >> 5] |= 1u << (j & 31);
  return ok();
}
}  // namespace

extern "C" {

int tac_make_signs(uint64_t seed, int layer, int kv, int d, uint32_t* out_words) {
  if (layer < 0) return fail(TAC_E_INVAL, "tac_make_signs: layer = %d", layer);
  if (kv != 0 && kv != 1) return fail(TAC_E_INVAL, "tac_make_signs: kv = %d (0 = K, 1 = V)", kv);
  return make_signs_q("tac_make_signs", seed, (uint64_t)(2 * (int64_t)layer + kv), d, out_words);
}

int tac_make_signs_shared(uint64_t seed, int d, uint32_t* out_words) {
  return make_signs_q("tac_make_signs_shared", seed, 0u, d, out_words);
}

int64_t tac_angle_row_bytes(const tac_layer_cfg* cfg) {
  if (check_cfg(cfg, "tac_angle_row_bytes")) return -1;
  return angle_row_bytes(cfg);
}

int64_t tac_norm_row_bytes(const tac_layer_cfg* cfg) {
  if (check_cfg(cfg, "tac_norm_row_bytes")) return -1;
  return norm_row_bytes(cfg);
}

int64_t tac_header_offset(const tac_layer_cfg* cfg, int64_t capacity) {
  if (check_cfg(cfg, "tac_header_offset") || capacity < 0) return -1;
  return header_offset(cfg, capacity);
}

int64_t tac_codes_bytes(const tac_layer_cfg* cfg, int64_t capacity) {
  if (check_cfg(cfg, "tac_codes_bytes") || capacity < 0) return -1;
  return capacity * angle_row_bytes(cfg);
}

int64_t tac_norms_bytes(const tac_layer_cfg* cfg, int64_t capacity) {
  if (check_cfg(cfg, "tac_norms_bytes") || capacity < 0) return -1;
  return header_offset(cfg, capacity) + (cfg->norm_mode == TAC_NORM_FP32 ? 0 : 8 * capacity);
}

double tac_avg_angle_bits(int num_layers, const int* n_k, const int* n_v) {
  if (num_layers <= 0 || !n_k || !n_v) return NAN;
  double acc = 0.0;
  for (int l = 0; l < num_layers; ++l) {
    if (n_k[l] < 1 || n_v[l] < 1) return NAN;
    acc += (std::log2((double)n_k[l]) + std::log2((double)n_v[l])) / 4.0;
  }
  return acc / (double)num_layers;
}

double tac_total_bits(double b_angle, double b_norm, int d) {
  if (d <= 0) return NAN;
  return b_angle + b_norm / 2.0 + 64.0 / (double)d;
}

int tac_rates(int num_layers, const int* n_k, const int* n_v, int b_k, int b_v, int d, double* out4) {
  static const char* who = "tac_rates";
  if (!out4) return fail(TAC_E_INVAL, "%s: out4 is NULL", who);
  if (num_layers <= 0 || !n_k || !n_v || d <= 0) return fail(TAC_E_INVAL, "%s: bad schedule", who);
  const bool fp32 = b_k == 32 && b_v == 32;
  if (!fp32 && (b_k < 1 || b_k > 16 || b_v < 1 || b_v > 16))
    return fail(TAC_E_INVAL, "%s: norm bits %d / %d (1..16, or 32 for fp32 norms)", who, b_k, b_v);
  const double angle = tac_avg_angle_bits(num_layers, n_k, n_v);
  if (std::isnan(angle)) return fail(TAC_E_INVAL, "%s: a codebook size is < 1", who);
  double stored = 0.0;
  for (int l = 0; l < num_layers; ++l) stored += tac::code_bits(n_k[l]) + tac::code_bits(n_v[l]);
  out4[0] = angle;                                   // Eq. 1
  out4[1] = angle + (b_k + b_v) / 4.0;               // payload: angle + norm bits per pair / 2
  out4[2] = fp32 ? out4[1] : tac_total_bits(angle, (b_k + b_v) / 2.0, d);   // Eq. 3
  out4[3] = stored / (4.0 * num_layers);             // bits the angle codes occupy
  return ok();
}

namespace {

// The kernel groups of one multi call are independent.  The first runs on the
// caller's stream, the others on library-owned streams (kSide per device,
// created on the first call that has several groups) that wait for the
// caller's stream at the call; the caller's stream waits for them before the
// call returns.  Small groups then fill the tail of the large one instead of
// queueing behind it, and the call stays ordered on the caller's stream
// (under stream capture this is the usual fork / join).
constexpr int kSide = 3;
struct SideStreams {
  bool init = false;
  cudaStream_t s[kSide] = {};
  cudaEvent_t fork = nullptr;
  cudaEvent_t join[kSide] = {};
};
std::mutex g_side_mu;
SideStreams g_side[64];

class GroupFork {
 public:
  GroupFork(cudaStream_t user, int ngroups) : user_(user) {
    if (ngroups <= 1) return;
    int dev = 0;
    if ((err_ = cudaGetDevice(&dev)) != cudaSuccess) return;
    if (dev < 0 || dev >= 64) { err_ = cudaErrorInvalidDevice; return; }
    lock_ = std::unique_lock<std::mutex>(g_side_mu);
    SideStreams& S = g_side[dev];
    if (!S.init) {
      for (int q = 0; q < kSide && err_ == cudaSuccess; ++q)
        if (!S.s[q]) err_ = cudaStreamCreateWithFlags(&S.s[q], cudaStreamNonBlocking);
      if (err_ == cudaSuccess && !S.fork) err_ = cudaEventCreateWithFlags(&S.fork, cudaEventDisableTiming);
      for (int q = 0; q < kSide && err_ == cudaSuccess; ++q)
        if (!S.join[q]) err_ = cudaEventCreateWithFlags(&S.join[q], cudaEventDisableTiming);
      if (err_ != cudaSuccess) return;
      S.init = true;
    }
    if ((err_ = cudaEventRecord(S.fork, user)) != cudaSuccess) return;
    st_ = &S;
  }
  cudaError_t error() const { return err_; }
  // Stream of group g (0 = the caller's).
  cudaStream_t stream(int g) {
    if (!st_ || g == 0) return user_;
    const int q = (g - 1) % kSide;
    if (q >= used_) {
      const cudaError_t e = cudaStreamWaitEvent(st_->s[q], st_->fork, 0);
      if (e != cudaSuccess && err_ == cudaSuccess) err_ = e;
      used_ = q + 1;
    }
    return st_->s[q];
  }
  // The caller's stream waits for every side stream used.
  cudaError_t join() {
    for (int q = 0; st_ && q < used_; ++q) {
      cudaError_t e = cudaEventRecord(st_->join[q], st_->s[q]);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(user_, st_->join[q], 0);
      if (e != cudaSuccess && err_ == cudaSuccess) err_ = e;
    }
    used_ = 0;
    return err_;
  }

 private:
  cudaStream_t user_;
  SideStreams* st_ = nullptr;
  std::unique_lock<std::mutex> lock_;
  int used_ = 0;
  cudaError_t err_ = cudaSuccess;
};

struct EncGroup {
  tac::EncParams p;
  int d, dt, na, nb, mode;
};
struct DecGroup {
  tac::DecParams p;
  int d, dt, na, nb, mode;
};

}  // namespace

namespace {

// Validates an encode call and groups its jobs by kernel: (d, dtype, n, norm
// bits, norm mode), one launch per group and up to TAC_MAX_JOBS jobs each,
// largest groups first.  Returns 0 or the call's tac status.
int plan_encode(const tac_encode_job* jobs, int njobs, const char* who, std::vector<EncGroup>& groups) {
  groups.clear();
  if (njobs < 0) return fail(TAC_E_INVAL, "%s: njobs = %d", who, njobs);
  if (njobs > 0 && !jobs) return fail(TAC_E_INVAL, "%s: jobs is NULL", who);
  // Validate everything before launching anything.
  std::vector<int> live;
  for (int j = 0; j < njobs; ++j) {
    const tac_encode_job& J = jobs[j];
    int rc = check_cfg(&J.cfg, who);
    if (rc) return rc;
    rc = check_rows(&J.x, J.cfg.d, who, "x");
    if (rc) return rc;
    if (J.capacity < 0) return fail(TAC_E_INVAL, "%s: job %d capacity < 0", who, j);
    if (J.x.rows == 0) continue;
    if (!J.codes || !J.norms) return fail(TAC_E_INVAL, "%s: job %d codes/norms is NULL", who, j);
    if (!aligned16(J.codes) || !aligned16(J.norms))
      return fail(TAC_E_INVAL, "%s: job %d codes/norms not 16-byte aligned", who, j);
    if (!J.slot && J.x.rows > J.capacity)
      return fail(TAC_E_INVAL, "%s: job %d rows %lld > capacity %lld", who, j, (long long)J.x.rows,
                  (long long)J.capacity);
    if (J.slot && ((uintptr_t)J.slot & 7u)) return fail(TAC_E_INVAL, "%s: job %d slot misaligned", who, j);
    if (J.status && ((uintptr_t)J.status & 3u)) return fail(TAC_E_INVAL, "%s: job %d status misaligned", who, j);
    live.push_back(j);
  }
  auto kernel_key = [&](int j) {
    const tac_encode_job& J = jobs[j];
    return (((J.cfg.d * 4 + J.x.dtype) * 512 + J.cfg.n_angle) * 64 + J.cfg.norm_bits) * 4 + J.cfg.norm_mode;
  };
  std::stable_sort(live.begin(), live.end(), [&](int a, int b) { return kernel_key(a) < kernel_key(b); });
  size_t i = 0;
  while (i < live.size()) {
    const int key = kernel_key(live[i]);
    const tac_layer_cfg& c0 = jobs[live[i]].cfg;
    const int d = c0.d, dt = jobs[live[i]].x.dtype;
    groups.emplace_back();
    EncGroup& G = groups.back();
    G.d = d; G.dt = dt; G.na = c0.n_angle; G.nb = c0.norm_bits; G.mode = c0.norm_mode;
    tac::EncParams& P = G.p;
    std::memset(&P, 0, sizeof(P));
    int64_t tiles = 0;
    while (i < live.size() && P.njobs < TAC_MAX_JOBS && kernel_key(live[i]) == key) {
      const tac_encode_job& J = jobs[live[i]];
      const int64_t tr = tile_rows(d);
      const int64_t jt = (J.x.rows + tr - 1) / tr;
      if (tiles + jt > 0x7fffffff / tr) break;          // warp-tile rows must index in 31 bits
      tac::EncJob& E = P.job[P.njobs];
      E.x = J.x.data;
      E.codes = static_cast<uint8_t*>(J.codes);
      E.norms = static_cast<uint8_t*>(J.norms);
      E.hdr = static_cast<uint8_t*>(J.norms) + header_offset(&J.cfg, J.capacity);
      E.slot = J.slot;
      E.status = J.status;
      E.capacity = J.capacity;
      E.rows = J.x.rows;
      E.stride = J.x.row_stride;
      copy_signs(E.signs, &J.cfg);
      E.w = tac::code_bits(J.cfg.n_angle);
      E.b = J.cfg.norm_bits;
      E.mode = J.cfg.norm_mode;
      E.tile0 = (int32_t)tiles;
      tiles += jt;
      ++P.njobs;
      ++i;
    }
    if (P.njobs == 0) return fail(TAC_E_UNSUPPORTED, "%s: a single job has too many rows", who);
    P.ntiles = (int32_t)tiles;
  }
  // largest groups first: the small ones fill the tail of the large ones
  std::stable_sort(groups.begin(), groups.end(),
                   [](const EncGroup& a, const EncGroup& b) { return a.p.ntiles > b.p.ntiles; });
  return 0;
}

// Workspace of an encode call: per launch group a 64-byte counter block and a
// bitmap of its warp-tile rows (together the part zeroed at the call), per
// group a copy of its job table (written by the encode kernel, read by the
// fix-up kernel), then per group its re-decision queue, 32-byte entries.  The queue's recommended
// capacity is one entry per 512 angle pairs plus 1024 (the synthetic caches
// of every workload queue about one per 2400 pairs); with less room the
// capacities shrink in proportion, down to none (then every row with a code to
// re-decide is re-decided whole through the bitmap).
constexpr int64_t kEncCtrBytes = 64, kEncEntryBytes = 32;
int64_t enc_ovf_bytes(const EncGroup& G) {
  const int64_t bits = (int64_t)G.p.ntiles * tile_rows(G.d);
  return ((bits + 127) / 128) * 16;
}
int64_t enc_job_bytes(const EncGroup& G) {
  return (((int64_t)G.p.njobs * (int64_t)sizeof(tac::EncJob) + 15) / 16) * 16;
}
int64_t enc_rec_cap(const EncGroup& G) {
  int64_t pairs = 0;
  for (int j = 0; j < G.p.njobs; ++j) pairs += G.p.job[j].rows * (G.d / 2);
  return pairs / 512 + 1024;
}
struct EncWs {
  int64_t zero = 0, jobs = 0, min = 0, rec = 0, rec_entries = 0;
};
EncWs enc_ws(const std::vector<EncGroup>& groups) {
  EncWs w;
  w.zero = kEncCtrBytes * (int64_t)groups.size();
  for (const EncGroup& G : groups) {
    w.zero += enc_ovf_bytes(G);
    w.jobs += enc_job_bytes(G);
    w.rec_entries += enc_rec_cap(G);
  }
  w.min = w.zero + w.jobs;
  w.rec = w.min + kEncEntryBytes * w.rec_entries;
  return w;
}

// Launches a planned encode call with its workspace (ws_bytes >= the minimum).
int run_encode(std::vector<EncGroup>& groups, uint8_t* ws, int64_t ws_bytes, cudaStream_t st, const char* who) {
  const int sms = num_sms();
  if (sms <= 0) return fail(TAC_E_CUDA, "%s: no CUDA device", who);
  const EncWs w = enc_ws(groups);
  const int64_t avail = (ws_bytes - w.min) / kEncEntryBytes;
  int64_t ovf_off = kEncCtrBytes * (int64_t)groups.size(), job_off = w.zero, q_off = w.min;
  for (size_t g = 0; g < groups.size(); ++g) {
    tac::EncParams& P = groups[g].p;
    const int64_t rc = enc_rec_cap(groups[g]);
    const int64_t cap = avail >= w.rec_entries ? rc : (int64_t)((double)rc * (double)avail / (double)w.rec_entries);
    P.gq_n = reinterpret_cast<unsigned long long*>(ws + kEncCtrBytes * (int64_t)g);
    P.ovf = reinterpret_cast<uint32_t*>(ws + ovf_off);
    P.gq = reinterpret_cast<uint4*>(ws + q_off);
    P.gq_cap = cap;
    P.gjobs = reinterpret_cast<tac::EncJob*>(ws + job_off);
    ovf_off += enc_ovf_bytes(groups[g]);
    job_off += enc_job_bytes(groups[g]);
    q_off += kEncEntryBytes * cap;
  }
  cudaError_t e = cudaMemsetAsync(ws, 0, (size_t)w.zero, st);
  if (e != cudaSuccess) return fail(TAC_E_CUDA, "%s: %s", who, cudaGetErrorString(e));
  static thread_local std::vector<int64_t> gtiles;
  static thread_local std::vector<int> caps;
  gtiles.resize(groups.size());
  caps.resize(groups.size());
  for (size_t g = 0; g < groups.size(); ++g) gtiles[g] = groups[g].p.ntiles;
  sm_shares(gtiles.data(), (int)groups.size(), sms, caps.data());
  // A call that gives every launch the whole GPU runs its encode launches
  // first and then all fix-ups side by side: an encode launch fills every SM,
  // so a fix-up queued behind it on its stream would not overlap the next
  // group's encode and the fix-ups would run one after another.  A small call
  // (launches on shares of the SMs, side by side) chains each group's fix-up
  // to its encode.
  bool whole = true;
  for (size_t g = 0; g < groups.size(); ++g) whole = whole && caps[g] == sms;
  const int rounds = whole && groups.size() > 1 ? 2 : 1;
  for (int r = 0; r < rounds; ++r) {
    const int phase = rounds == 1 ? 3 : r + 1;
    GroupFork fork(st, (int)groups.size());
    if (fork.error() != cudaSuccess) return fail(TAC_E_CUDA, "%s: %s", who, cudaGetErrorString(fork.error()));
    for (size_t g = 0; g < groups.size(); ++g) {
      const EncGroup& G = groups[g];
      e = tac::launch_encode(G.d, G.dt, G.na, G.nb, G.mode, G.p, caps[g], fork.stream((int)g), phase);
      if (e != cudaSuccess) {
        fork.join();
        return fail(TAC_E_CUDA, "%s: launch failed: %s", who, cudaGetErrorString(e));
      }
    }
    e = fork.join();
    if (e != cudaSuccess) return fail(TAC_E_CUDA, "%s: %s", who, cudaGetErrorString(e));
  }
  return 0;
}

}  // namespace

int64_t tac_encode_workspace_bytes(const tac_encode_job* jobs, int njobs, int64_t* min_bytes) {
  static thread_local std::vector<EncGroup> groups;
  if (plan_encode(jobs, njobs, "tac_encode_workspace_bytes", groups)) return -1;
  const EncWs w = enc_ws(groups);
  if (min_bytes) *min_bytes = w.min;
  ok();
  return w.rec;
}

int tac_encode_multi_ws(const tac_encode_job* jobs, int njobs, void* workspace, int64_t workspace_bytes,
                        tac_stream_t stream) {
  static const char* who = "tac_encode_multi_ws";
  static thread_local std::vector<EncGroup> groups;
  int rc = plan_encode(jobs, njobs, who, groups);
  if (rc) return rc;
  if (groups.empty()) return ok();
  const EncWs w = enc_ws(groups);
  if (!workspace || !aligned16(workspace)) return fail(TAC_E_INVAL, "%s: workspace NULL or not 16-byte aligned", who);
  if (workspace_bytes < w.min)
    return fail(TAC_E_INVAL, "%s: workspace of %lld bytes < the minimum %lld", who, (long long)workspace_bytes,
                (long long)w.min);
  rc = run_encode(groups, static_cast<uint8_t*>(workspace), workspace_bytes, reinterpret_cast<cudaStream_t>(stream),
                  who);
  return rc ? rc : ok();
}

int tac_encode_multi(const tac_encode_job* jobs, int njobs, tac_stream_t stream) {
  static const char* who = "tac_encode_multi";
  static thread_local std::vector<EncGroup> groups;
  int rc = plan_encode(jobs, njobs, who, groups);
  if (rc) return rc;
  if (groups.empty()) return ok();
  const EncWs w = enc_ws(groups);
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  void* ws = nullptr;
  cudaError_t e = cudaMallocAsync(&ws, (size_t)w.rec, st);
  if (e != cudaSuccess) return fail(TAC_E_CUDA, "%s: workspace allocation: %s", who, cudaGetErrorString(e));
  rc = run_encode(groups, static_cast<uint8_t*>(ws), w.rec, st, who);
  e = cudaFreeAsync(ws, st);
  if (rc) return rc;
  if (e != cudaSuccess) return fail(TAC_E_CUDA, "%s: %s", who, cudaGetErrorString(e));
  return ok();
}

int tac_decode_multi(const tac_decode_job* jobs, int njobs, tac_stream_t stream) {
  static const char* who = "tac_decode_multi";
  if (njobs < 0) return fail(TAC_E_INVAL, "%s: njobs = %d", who, njobs);
  if (njobs > 0 && !jobs) return fail(TAC_E_INVAL, "%s: jobs is NULL", who);
  std::vector<int> live;
  for (int j = 0; j < njobs; ++j) {
    const tac_decode_job& J = jobs[j];
    int rc = check_cfg(&J.cfg, who);
    if (rc) return rc;
    rc = check_rows(&J.y, J.cfg.d, who, "y");
    if (rc) return rc;
    if (J.capacity < 0) return fail(TAC_E_INVAL, "%s: job %d capacity < 0", who, j);
    if (J.y.rows == 0) continue;
    if (!J.codes || !J.norms) return fail(TAC_E_INVAL, "%s: job %d codes/norms is NULL", who, j);
    if (!aligned16(J.codes) || !aligned16(J.norms))
      return fail(TAC_E_INVAL, "%s: job %d codes/norms not 16-byte aligned", who, j);
    if (!J.slot && J.y.rows > J.capacity)
      return fail(TAC_E_INVAL, "%s: job %d rows %lld > capacity %lld", who, j, (long long)J.y.rows,
                  (long long)J.capacity);
    if (J.slot && ((uintptr_t)J.slot & 7u)) return fail(TAC_E_INVAL, "%s: job %d slot misaligned", who, j);
    live.push_back(j);
  }
  const int sms = num_sms();
  if (live.empty()) return ok();
  if (sms <= 0) return fail(TAC_E_CUDA, "%s: no CUDA device", who);
  // Group by kernel: (d, dtype, n, norm bits, norm mode); one launch per group
  // and up to TAC_MAX_JOBS jobs per launch.
  auto kernel_key = [&](int j) {
    const tac_decode_job& J = jobs[j];
    return (((J.cfg.d * 4 + J.y.dtype) * 512 + J.cfg.n_angle) * 64 + J.cfg.norm_bits) * 4 + J.cfg.norm_mode;
  };
  std::stable_sort(live.begin(), live.end(), [&](int a, int b) { return kernel_key(a) < kernel_key(b); });
  static thread_local std::vector<DecGroup> groups;
  groups.clear();
  size_t i = 0;
  while (i < live.size()) {
    const int key = kernel_key(live[i]);
    const tac_layer_cfg& c0 = jobs[live[i]].cfg;
    const int d = c0.d, dt = jobs[live[i]].y.dtype;
    const int na = c0.n_angle, nb = c0.norm_bits, mode = c0.norm_mode;
    groups.emplace_back();
    DecGroup& G = groups.back();
    G.d = d; G.dt = dt; G.na = na; G.nb = nb; G.mode = mode;
    tac::DecParams& P = G.p;
    std::memset(&P, 0, sizeof(P));
    int64_t tiles = 0;
    while (i < live.size() && P.njobs < TAC_MAX_JOBS && kernel_key(live[i]) == key) {
      const tac_decode_job& J = jobs[live[i]];
      const int64_t tr = tile_rows(d);
      const int64_t jt = (J.y.rows + tr - 1) / tr;
      if (tiles + jt > 0x7fffffff) break;
      tac::DecJob& E = P.job[P.njobs];
      E.codes = static_cast<const uint8_t*>(J.codes);
      E.norms = static_cast<const uint8_t*>(J.norms);
      E.hdr = static_cast<const uint8_t*>(J.norms) + header_offset(&J.cfg, J.capacity);
      E.slot = J.slot;
      E.capacity = J.capacity;
      E.y = J.y.data;
      E.rows = J.y.rows;
      E.stride = J.y.row_stride;
      copy_signs(E.signs, &J.cfg);
      E.w = tac::code_bits(J.cfg.n_angle);
      E.b = J.cfg.norm_bits;
      E.mode = J.cfg.norm_mode;
      E.tile0 = (int32_t)tiles;
      tiles += jt;
      ++P.njobs;
      ++i;
    }
    if (P.njobs == 0) return fail(TAC_E_UNSUPPORTED, "%s: a single job has too many rows", who);
    P.ntiles = (int32_t)tiles;
  }
  std::stable_sort(groups.begin(), groups.end(),
                   [](const DecGroup& a, const DecGroup& b) { return a.p.ntiles > b.p.ntiles; });
  static thread_local std::vector<int64_t> gtiles;
  static thread_local std::vector<int> caps;
  gtiles.resize(groups.size());
  caps.resize(groups.size());
  for (size_t g = 0; g < groups.size(); ++g) gtiles[g] = groups[g].p.ntiles;
  sm_shares(gtiles.data(), (int)groups.size(), sms, caps.data());
  GroupFork fork(reinterpret_cast<cudaStream_t>(stream), (int)groups.size());
  if (fork.error() != cudaSuccess) return fail(TAC_E_CUDA, "%s: %s", who, cudaGetErrorString(fork.error()));
  for (size_t g = 0; g < groups.size(); ++g) {
    const DecGroup& G = groups[g];
    cudaError_t e = tac::launch_decode(G.d, G.dt, G.na, G.nb, G.mode, G.p, caps[g], fork.stream((int)g));
    if (e != cudaSuccess) {
      fork.join();
      return fail(TAC_E_CUDA, "%s: launch failed: %s", who, cudaGetErrorString(e));
    }
  }
  const cudaError_t e = fork.join();
  if (e != cudaSuccess) return fail(TAC_E_CUDA, "%s: %s", who, cudaGetErrorString(e));
  return ok();
}

int tac_encode(const tac_rows* x, const tac_layer_cfg* cfg, void* out_codes, void* out_norms,
               tac_stream_t stream) {
  if (!x) return fail(TAC_E_INVAL, "tac_encode: x is NULL");
  if (!cfg) return fail(TAC_E_INVAL, "tac_encode: cfg is NULL");
  tac_encode_job j;
  std::memset(&j, 0, sizeof(j));
  j.cfg = *cfg;
  j.x = *x;
  j.codes = out_codes;
  j.norms = out_norms;
  j.capacity = x->rows;
  j.slot = nullptr;
  return tac_encode_multi(&j, 1, stream);
}

int tac_encode_checked(const tac_rows* x, const tac_layer_cfg* cfg, void* out_codes, void* out_norms,
                       uint32_t* status, tac_stream_t stream) {
  if (!x) return fail(TAC_E_INVAL, "tac_encode_checked: x is NULL");
  if (!cfg) return fail(TAC_E_INVAL, "tac_encode_checked: cfg is NULL");
  if (!status) return fail(TAC_E_INVAL, "tac_encode_checked: status is NULL");
  tac_encode_job j;
  std::memset(&j, 0, sizeof(j));
  j.cfg = *cfg;
  j.x = *x;
  j.codes = out_codes;
  j.norms = out_norms;
  j.capacity = x->rows;
  j.slot = nullptr;
  j.status = status;
  return tac_encode_multi(&j, 1, stream);
}

int tac_decode(const void* codes, const void* norms, const tac_layer_cfg* cfg, tac_rows* y,
               tac_stream_t stream) {
  if (!y) return fail(TAC_E_INVAL, "tac_decode: y is NULL");
  if (!cfg) return fail(TAC_E_INVAL, "tac_decode: cfg is NULL");
  tac_decode_job j;
  std::memset(&j, 0, sizeof(j));
  j.cfg = *cfg;
  j.codes = codes;
  j.norms = norms;
  j.capacity = y->rows;
  j.slot = nullptr;
  j.y = *y;
  return tac_decode_multi(&j, 1, stream);
}

// ---------------------------------------------------------------------------
// Attention from records
// ---------------------------------------------------------------------------
namespace {

int check_attend_job(const tac_attend_job& J, int j, const char* who) {
  int rc = check_cfg(&J.cfg_k, who);
  if (rc) return rc;
  rc = check_cfg(&J.cfg_v, who);
  if (rc) return rc;
  const int d = J.cfg_k.d;
  if (J.cfg_v.d != d) return fail(TAC_E_INVAL, "%s: job %d K and V d differ (%d, %d)", who, j, d, J.cfg_v.d);
  if (d != 64 && d != 128) return fail(TAC_E_UNSUPPORTED, "%s: job %d d = %d (64, 128)", who, j, d);
  rc = check_rows(&J.q, d, who, "q");
  if (rc) return rc;
  rc = check_rows(&J.out, d, who, "out");
  if (rc) return rc;
  if (J.q.rows < 1 || J.q.rows > TAC_MAX_QUERIES)
    return fail(TAC_E_INVAL, "%s: job %d has %lld query rows (1..%d)", who, j, (long long)J.q.rows, TAC_MAX_QUERIES);
  if (J.out.rows != J.q.rows || J.out.dtype != J.q.dtype)
    return fail(TAC_E_INVAL, "%s: job %d out must match q in rows and dtype", who, j);
  if (J.tokens < 1 || J.tokens > J.capacity)
    return fail(TAC_E_INVAL, "%s: job %d tokens %lld outside 1..capacity %lld", who, j, (long long)J.tokens,
                (long long)J.capacity);
  if ((J.tokens + TAC_ATTEND_SPLIT - 1) / TAC_ATTEND_SPLIT > (1 << 26))
    return fail(TAC_E_UNSUPPORTED, "%s: job %d tokens %lld too many", who, j, (long long)J.tokens);
  if (!J.k_codes || !J.k_norms || !J.v_codes || !J.v_norms)
    return fail(TAC_E_INVAL, "%s: job %d record plane is NULL", who, j);
  if (!aligned16(J.k_codes) || !aligned16(J.k_norms) || !aligned16(J.v_codes) || !aligned16(J.v_norms))
    return fail(TAC_E_INVAL, "%s: job %d record planes not 16-byte aligned", who, j);
  if (!(J.scale == J.scale)) return fail(TAC_E_INVAL, "%s: job %d scale is NaN", who, j);
  return TAC_OK;
}

int64_t attend_ws_floats(const tac_attend_job& J) {
  const int64_t splits = (J.tokens + TAC_ATTEND_SPLIT - 1) / TAC_ATTEND_SPLIT;
  const int64_t f = splits * J.q.rows * tac::att_rec_floats(J.cfg_k.d);
  return (f + 3) & ~(int64_t)3;  // 16-byte multiple
}

}  // namespace

int64_t tac_attend_workspace_bytes(const tac_attend_job* jobs, int njobs) {
  static const char* who = "tac_attend_workspace_bytes";
  if (njobs < 0 || (njobs > 0 && !jobs)) { fail(TAC_E_INVAL, "%s: bad job array", who); return -1; }
  int64_t f = 0;
  for (int j = 0; j < njobs; ++j) {
    if (check_attend_job(jobs[j], j, who)) return -1;
    f += attend_ws_floats(jobs[j]);
  }
  ok();
  return 4 * f;
}

namespace {

// Validates the jobs; *need = the workspace bytes they take.
int check_attend_jobs(const tac_attend_job* jobs, int njobs, int64_t* need, const char* who) {
  if (njobs < 0) return fail(TAC_E_INVAL, "%s: njobs = %d", who, njobs);
  if (njobs > 0 && !jobs) return fail(TAC_E_INVAL, "%s: jobs is NULL", who);
  *need = 0;
  for (int j = 0; j < njobs; ++j) {
    const int rc = check_attend_job(jobs[j], j, who);
    if (rc) return rc;
    *need += 4 * attend_ws_floats(jobs[j]);
  }
  return TAC_OK;
}

// Launches checked jobs, grouped by (d, dtype) in job order, up to
// TAC_ATTEND_MAX_JOBS per launch pair; each job's workspace part follows the
// previous one's.  `concurrent`: several launch pairs run concurrently
// (GroupFork); otherwise back to back on `st`.  Allocates nothing.
int run_attend(const tac_attend_job* jobs, int njobs, float* ws, cudaStream_t st, bool concurrent, const char* who) {
  static_assert(sizeof(tac::AttParams) <= 32764, "kernel parameter limit");
  static thread_local tac::AttParams P;
  static const int kD[2] = {64, 128};
  static const int kDt[2] = {TAC_BF16, TAC_FP32};
  int ngroups = 0;
  for (int d : kD)
    for (int dt : kDt) {
      int c = 0;
      for (int j = 0; j < njobs; ++j) c += jobs[j].cfg_k.d == d && jobs[j].q.dtype == dt;
      ngroups += (c + TAC_ATTEND_MAX_JOBS - 1) / TAC_ATTEND_MAX_JOBS;
    }
  GroupFork fork(st, concurrent ? ngroups : 1);
  if (fork.error() != cudaSuccess) return fail(TAC_E_CUDA, "%s: %s", who, cudaGetErrorString(fork.error()));
  int g = 0;
  int64_t ws_off = 0;
  for (int d : kD) {
    for (int dt : kDt) {
      int i = 0;
      auto next = [&](int from) {
        while (from < njobs && !(jobs[from].cfg_k.d == d && jobs[from].q.dtype == dt)) ++from;
        return from;
      };
      i = next(0);
      while (i < njobs) {
        std::memset(&P, 0, sizeof(P));
        int64_t splits = 0;
        int nrows = 0, nq_max = 1;
        while (i < njobs && P.njobs < TAC_ATTEND_MAX_JOBS) {
          const tac_attend_job& J = jobs[i];
          const int64_t ns = (J.tokens + TAC_ATTEND_SPLIT - 1) / TAC_ATTEND_SPLIT;
          if (splits + ns > 0x7fffffff) break;   // CTAs (<= splits) are assigned at launch
          tac::AttJob& A = P.job[P.njobs];
          A.kc = static_cast<const uint8_t*>(J.k_codes);
          A.kn = static_cast<const uint8_t*>(J.k_norms);
          A.kh = A.kn + header_offset(&J.cfg_k, J.capacity);
          A.vc = static_cast<const uint8_t*>(J.v_codes);
          A.vn = static_cast<const uint8_t*>(J.v_norms);
          A.vh = A.vn + header_offset(&J.cfg_v, J.capacity);
          A.q = J.q.data;
          A.out = J.out.data;
          A.q_stride = J.q.row_stride;
          A.out_stride = J.out.row_stride;
          A.tokens = J.tokens;
          A.scale = J.scale;
          A.nq = (int32_t)J.q.rows;
          A.nk = J.cfg_k.n_angle; A.wk = tac::code_bits(J.cfg_k.n_angle); A.bk = J.cfg_k.norm_bits; A.mk = J.cfg_k.norm_mode;
          A.nv = J.cfg_v.n_angle; A.wv = tac::code_bits(J.cfg_v.n_angle); A.bv = J.cfg_v.norm_bits; A.mv = J.cfg_v.norm_mode;
          A.inv_lk = A.mk == TAC_NORM_FP32 ? 0.f : 1.f / (float)((1 << A.bk) - 1);
          A.inv_lv = A.mv == TAC_NORM_FP32 ? 0.f : 1.f / (float)((1 << A.bv) - 1);
          A.lgrk = tac::att_table_lgr(1 << A.wk);
          A.lgrv = tac::att_table_lgr(1 << A.wv);
          A.ck = tac::att_norm_case(A.bk, A.mk);
          A.cv = tac::att_norm_case(A.bv, A.mv);
          copy_signs(A.sk, &J.cfg_k);
          copy_signs(A.sv, &J.cfg_v);
          A.split0 = (int32_t)splits;
          A.ws = ws_off;
          ws_off += attend_ws_floats(J);
          splits += ns;
          nrows += A.nq;
          nq_max = std::max(nq_max, (int)A.nq);
          ++P.njobs;
          i = next(i + 1);
        }
        if (P.njobs == 0) {
          fork.join();
          return fail(TAC_E_UNSUPPORTED, "%s: a single job has too many tokens", who);
        }
        P.nsplits = (int32_t)splits;
        P.q_bf16 = dt == TAC_BF16;
        cudaError_t e = tac::launch_attend(d, dt, nq_max, P, nrows, ws, fork.stream(g++));
        if (e != cudaSuccess) {
          fork.join();
          return fail(TAC_E_CUDA, "%s: launch failed: %s", who, cudaGetErrorString(e));
        }
      }
    }
  }
  const cudaError_t e = fork.join();
  if (e != cudaSuccess) return fail(TAC_E_CUDA, "%s: %s", who, cudaGetErrorString(e));
  return ok();
}

}  // namespace

int tac_attend_multi(const tac_attend_job* jobs, int njobs, void* workspace, int64_t workspace_bytes,
                     tac_stream_t stream) {
  static const char* who = "tac_attend_multi";
  int64_t need = 0;
  const int rc = check_attend_jobs(jobs, njobs, &need, who);
  if (rc) return rc;
  if (njobs == 0) return ok();
  if (!workspace || !aligned16(workspace) || workspace_bytes < need)
    return fail(TAC_E_INVAL, "%s: workspace NULL, misaligned or smaller than %lld bytes", who, (long long)need);
  if (num_sms() <= 0) return fail(TAC_E_CUDA, "%s: no CUDA device", who);
  return run_attend(jobs, njobs, static_cast<float*>(workspace), reinterpret_cast<cudaStream_t>(stream), true, who);
}

int tac_attend_multi_static(const tac_attend_job* jobs, int njobs, tac_stream_t stream) {
  static const char* who = "tac_attend_multi_static";
  int64_t need = 0;
  const int rc = check_attend_jobs(jobs, njobs, &need, who);
  if (rc) return rc;
  if (need > TAC_ATTEND_STATIC_WS_BYTES)
    return fail(TAC_E_UNSUPPORTED,
                "%s: these jobs need %lld bytes of workspace, the static workspace holds %lld; "
                "split them over several calls or use tac_attend_multi",
                who, (long long)need, (long long)TAC_ATTEND_STATIC_WS_BYTES);
  float* ws = nullptr;
  const cudaError_t e = tac::attend_static_workspace(&ws);
  if (e != cudaSuccess) return fail(TAC_E_CUDA, "%s: static workspace: %s", who, cudaGetErrorString(e));
  if (num_sms() <= 0) return fail(TAC_E_CUDA, "%s: no CUDA device", who);   // cached for later calls
  if (njobs == 0) return ok();
  return run_attend(jobs, njobs, ws, reinterpret_cast<cudaStream_t>(stream), false, who);
}

int tac_fwht_debug(const tac_rows* x, int d, const uint32_t* signs, float* y, tac_stream_t stream) {
  static const char* who = "tac_fwht_debug";
  if (d < 2 || d > 128 || (d & (d - 1))) return fail(TAC_E_INVAL, "%s: d = %d (powers of two 2..128)", who, d);
  if (!signs) return fail(TAC_E_INVAL, "%s: signs is NULL", who);
  int rc = check_rows(x, d, who, "x", /*rows16=*/false);
  if (rc) return rc;
  if (x->rows == 0) return ok();
  if (!y || !aligned16(y)) return fail(TAC_E_INVAL, "%s: y is NULL or misaligned", who);
  if (num_sms() <= 0) return fail(TAC_E_CUDA, "%s: no CUDA device", who);
  uint32_t s[4] = {0, 0, 0, 0};
  for (int q = 0; q < (d + 31) / 32; ++q) s[q] = signs[q];
  if (d < 32) s[0] &= (1u << d) - 1u;
  cudaError_t e = tac::launch_fwht_debug(d, x->data, x->dtype, x->rows, x->row_stride, s, y,
                                         reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail(TAC_E_CUDA, "%s: launch failed: %s", who, cudaGetErrorString(e));
  return ok();
}

int tac_hw_approx_debug(int op, const float* x, float* y, int64_t n, tac_stream_t stream) {
  static const char* who = "tac_hw_approx_debug";
  if (op < 0 || op > 5) return fail(TAC_E_INVAL, "%s: op = %d (0..5)", who, op);
  if (n < 0) return fail(TAC_E_INVAL, "%s: n = %lld", who, (long long)n);
  if (n == 0) return ok();
  if (!x || !y || !aligned16(x) || !aligned16(y)) return fail(TAC_E_INVAL, "%s: x or y is NULL or misaligned", who);
  const int sms = num_sms();
  if (sms <= 0) return fail(TAC_E_CUDA, "%s: no CUDA device", who);
  cudaError_t e = tac::launch_hw_approx(op, x, y, n, sms, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail(TAC_E_CUDA, "%s: launch failed: %s", who, cudaGetErrorString(e));
  return ok();
}

}  // extern "C"
