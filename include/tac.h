/*
 * tac.h -- C ABI of libtac, a GB300 (sm_103a) implementation of the TurboAngle
 * KV-cache encode/decode path (arXiv 2603.27467, "TurboAngle: Near-Lossless KV
 * Cache Compression via Uniform Angle Quantization").
 *
 * What the library computes, per head vector x of dimension d (one "row"):
 *   encode (Alg. 1 with Sec. 3.3):
 *     y = H D x                 D: random +-1 diagonal, H: normalized Hadamard (Sec. 2)
 *     r_i = |(y_2i, y_2i+1)|, theta_i = atan2(y_2i+1, y_2i)          (Alg. 1)
 *     k_i = floor(n theta_i / 2 pi + 1/2) mod n                      (Alg. 1)
 *     c_i = round((r_i - r_min)/(r_max - r_min) (2^b - 1))           (Eq. 2, linear)
 *           or Eq. 2 applied to log2 r_i                              (Sec. 3.3, log-space)
 *     stored: k_i (ceil(log2 n) bits each), c_i (b bits each), (r_min, r_max) as fp32;
 *     or, with TAC_NORM_FP32 (the angle-only configuration of Sec. 3.1 / Tables 1-4),
 *     r_i itself as fp32 (b = 32) and no (r_min, r_max).
 *   decode (Sec. 3.1): y^_2i = r^_i cos(2 pi k_i / n), y^_2i+1 = r^_i sin(2 pi k_i / n),
 *     x^ = D H y^, with r^_i the dequantized norm (r_min + c (r_max - r_min)/(2^b - 1), or
 *     the same in log2 space).
 *
 * Record layout ("three planes", caller-owned device memory, one record slot per row):
 *   angle plane   slot s at  codes + s * tac_angle_row_bytes(cfg):  d/2 codes of w = ceil(log2 n)
 *                 bits, one LSB-first bitstream per row (the code in position v occupies bits
 *                 [v*w, v*w + w)).  Position v holds the code of pair i = phi(v):
 *                   d = 64, 128 (L = d/16):  phi(v) = 4 (v mod L) + ((v / L) mod 4) + 4 L floor(v / 4L)
 *                   d = 16, 32:              phi(v) = v
 *                 (pair i = elements 2i, 2i+1 of the transformed row).  The order lets a kernel
 *                 that splits a row over L lanes of 8 positions move two runs of 4 consecutive
 *                 pairs per lane; the paper fixes no layout.
 *   norm plane    slot s at  norms + s * tac_norm_row_bytes(cfg):   d/2 codes of b bits, same
 *                 positions (TAC_NORM_FP32: d/2 little-endian floats, position v = r_phi(v)).
 *   header plane  slot s at  norms + tac_header_offset(cfg, capacity) + 8*s:
 *                 float r_min, float r_max (little endian); absent with TAC_NORM_FP32.
 *
 * Conventions shared by every entry point:
 *   - All device pointers must be 16-byte aligned; rows are row_stride elements
 *     apart and row_stride * sizeof(element) must be a multiple of 16.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and never synchronize (the batched calls create their helper
 *     streams once, see tac_encode_multi).  They allocate no device memory,
 *     except that tac_encode, tac_encode_checked and tac_encode_multi take the
 *     encode's re-decision workspace from the device's stream-ordered memory
 *     pool (cudaMallocAsync / cudaFreeAsync on `stream`); tac_encode_multi_ws
 *     takes it from the caller instead.
 *   - Errors: a nonzero tac_status is returned and tac_last_error() gives a message
 *     (per host thread).  TAC_E_INVAL: a bad argument (nothing launched).
 *     TAC_E_UNSUPPORTED: a valid but unimplemented shape (nothing launched).
 *     TAC_E_CUDA: the launch failed (cudaGetLastError after the launch).
 *   - Inputs must be finite with |x_j| <= 2^56, and each nonzero |x_j| >= 2^-53
 *     for bf16 rows (>= 2^-37 for fp32 rows): then every nonzero pair energy
 *     E^2 + O^2 of the butterfly is a normal fp32 number and the codes and header
 *     match the definitions within the stated tolerances.  A row holding a NaN
 *     or an infinity gets a defined record instead: every angle and norm code 0
 *     and the header (NaN, NaN) (with fp32 norms: every norm NaN), which decodes
 *     to a NaN row; an encode given a status word (tac_encode_checked, or the
 *     status field of a tac_encode_job) stores TAC_E_NONFINITE in it.  Finite
 *     values outside the range give unspecified codes but never out-of-bounds
 *     accesses.
 */
#ifndef TAC_H_
#define TAC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* tac_stream_t; /* == cudaStream_t */

typedef enum {
  TAC_OK = 0,
  TAC_E_INVAL = 1,
  TAC_E_UNSUPPORTED = 2,
  TAC_E_CUDA = 3,
  TAC_E_NONFINITE = 4   /* written (asynchronously) to an encode's status word: a row held a NaN or an inf */
} tac_status;

/* Norm storage: Eq. 2 linear, Eq. 2 on log2 r (Sec. 3.3), or the pair norms as fp32
 * (Sec. 3.1: "each pair norm r_i is stored in fp32"; norm_bits must be 32). */
typedef enum { TAC_NORM_LINEAR = 0, TAC_NORM_LOG = 1, TAC_NORM_FP32 = 2 } tac_norm_mode;
typedef enum { TAC_BF16 = 0, TAC_FP32 = 1 } tac_dtype;

#define TAC_MAX_D 128
#define TAC_MAX_JOBS 96

/*
 * One codebook: the quantizer of one (layer, K or V) cache (Sec. 3.2 assigns an
 * independent (n_K, n_V) per layer; Sec. 3.3 picks the norm bits/mode per K/V).
 * Plain host struct, passed by pointer and copied at each call.
 */
typedef struct {
  int32_t d;          /* head dimension: 16, 32, 64 or 128 */
  int32_t n_angle;    /* angle bins n: a power of two 2..256, or 48 or 56 (Table 1) */
  int32_t norm_bits;  /* b: 4 or 8 (linear / log), 32 (TAC_NORM_FP32) */
  int32_t norm_mode;  /* tac_norm_mode */
  uint32_t signs[TAC_MAX_D / 32]; /* D: bit j of the little-endian word array set <=> s_j = -1
                                     (from tac_make_signs); bits >= d are ignored */
} tac_layer_cfg;

/* A block of rows: `rows` vectors of cfg.d elements, row i at data + i*row_stride elements. */
typedef struct {
  void* data;           /* device pointer */
  int32_t dtype;        /* tac_dtype */
  int64_t rows;         /* >= 0 */
  int64_t row_stride;   /* elements, >= d */
} tac_rows;

/* One encode job of a batched launch: rows of x -> record slots (scatter-append). */
typedef struct {
  tac_layer_cfg cfg;
  tac_rows x;            /* input rows (device) */
  void* codes;           /* angle plane of the destination cache (device) */
  void* norms;           /* norm + header planes of the destination cache (device) */
  int64_t capacity;      /* record slots in the destination planes */
  const int64_t* slot;   /* device, x.rows entries: destination slot of row i, each in
                            [0, capacity); NULL means slot i (then x.rows <= capacity).
                            Duplicate slots race (one of the writers wins). */
  uint32_t* status;      /* device, 4-byte aligned, or NULL: TAC_E_NONFINITE is stored in
                            it when a row of x holds a NaN or an infinity; otherwise it is
                            left as it is (the caller zeroes it; jobs may share one) */
} tac_encode_job;

/* One decode job of a batched launch: record slots -> rows of y (gather). */
typedef struct {
  tac_layer_cfg cfg;
  const void* codes;     /* angle plane of the source cache (device) */
  const void* norms;     /* norm + header planes of the source cache (device) */
  int64_t capacity;      /* record slots in the source planes */
  const int64_t* slot;   /* device, y.rows entries: source slot of output row i; a slot
                            outside [0, capacity) decodes as an all-zero record (the
                            row r_min = r_max = 0: zeros); NULL means slot i */
  tac_rows y;            /* output rows (device), bf16 (round to nearest even) or fp32 */
} tac_decode_job;

/*
 * D of Sec. 2 ("s_i ~ Uniform{+1,-1}", sampled once from a seeded PRNG, Sec. 3.1
 * implementation note), one per (layer, K/V).  Counter-based SplitMix64
 * (Steele, Lea, Flood 2014):
 *   key = output #q of the SplitMix64 stream seeded with `seed`, q = 2*layer + kv;
 *   s_j = -1 iff bit 63 of output #j of the stream seeded with key is set.
 * Output #i of the stream seeded with z is mix(z + (i+1)*0x9E3779B97F4A7C15).
 * Writes ceil(d/32) words (host memory; bit j of the little-endian word array
 * set <=> s_j = -1).  kv: 0 = K, 1 = V.  Host only; TAC_E_INVAL for a NULL
 * out_words, d outside 1..2^20, layer < 0 or kv not 0/1.
 */
int tac_make_signs(uint64_t seed, int layer, int kv, int d, uint32_t* out_words);

/* The paper's single D for every layer and K/V (Sec. 3.1 implementation note):
 * the stream keyed by output #0, i.e. tac_make_signs' q = 0. */
int tac_make_signs_shared(uint64_t seed, int d, uint32_t* out_words);

/* Bytes per row of each plane (Sec. 3.1 rate: log2(n) bits per pair, stored in
 * ceil(log2 n) bits; Eq. 3 norm bits per pair; 64 bits of header per vector).
 * Return -1 for an invalid cfg. */
int64_t tac_angle_row_bytes(const tac_layer_cfg* cfg);   /* d/2 * ceil(log2 n) / 8 */
int64_t tac_norm_row_bytes(const tac_layer_cfg* cfg);    /* d/2 * b / 8 */
/* Byte offset of the header plane inside `norms` for a cache of `capacity` slots:
 * capacity * tac_norm_row_bytes rounded up to a multiple of 16. */
int64_t tac_header_offset(const tac_layer_cfg* cfg, int64_t capacity);
int64_t tac_codes_bytes(const tac_layer_cfg* cfg, int64_t capacity); /* angle plane size */
/* norm + header planes: tac_header_offset + 8 * capacity (no header with TAC_NORM_FP32) */
int64_t tac_norms_bytes(const tac_layer_cfg* cfg, int64_t capacity);

/* Eq. 1: (1/L) sum_l (log2 n_K^l + log2 n_V^l) / 4.  Returns NaN if an n is < 1. */
double tac_avg_angle_bits(int num_layers, const int* n_k, const int* n_v);
/* Eq. 3: b_angle + b_norm / 2 + 64 / d. */
double tac_total_bits(double b_angle, double b_norm, int d);

/*
 * Rates of a per-layer schedule (n_k[l], n_v[l]) with norm bits b_k, b_v
 * (Sec. 3.2, 3.3), written to out4 (host, 4 doubles):
 *   [0] Eq. 1 angle bits per element;
 *   [1] payload bits per element: [0] + (b_k + b_v) / 4 (norm bits per pair / 2,
 *       averaged over K and V);
 *   [2] Eq. 3 total: [0] + (b_k + b_v) / 4 + 64/d; with fp32 norms
 *       (b_k = b_v = 32, Sec. 3.1) the payload itself (no min/max header);
 *   [3] bits the angle codes occupy: ceil(log2 n) instead of log2 n.
 * TAC_E_INVAL for a bad schedule (num_layers < 1, an n < 1, d < 1, norm bits
 * outside 1..16 unless both are 32).
 */
int tac_rates(int num_layers, const int* n_k, const int* n_v, int b_k, int b_v, int d, double* out4);

/*
 * Encode x.rows rows (Alg. 1 + Eq. 2) into record slots 0..x.rows-1 of
 * (out_codes, out_norms), a cache of capacity x.rows
 * (sizes: tac_codes_bytes(cfg, x.rows), tac_norms_bytes(cfg, x.rows)).
 */
int tac_encode(const tac_rows* x, const tac_layer_cfg* cfg, void* out_codes, void* out_norms,
               tac_stream_t stream);

/*
 * tac_encode with a status word (device, 4-byte aligned, zeroed by the caller):
 * TAC_E_NONFINITE is stored in *status, in stream order, when a row of x holds a
 * NaN or an infinity (the paper fixes no behaviour for them; this library's
 * records for such rows are described under the conventions above).  The
 * return value reports argument and launch errors only, as for tac_encode.
 */
int tac_encode_checked(const tac_rows* x, const tac_layer_cfg* cfg, void* out_codes, void* out_norms,
                       uint32_t* status, tac_stream_t stream);

/*
 * Decode y->rows records (slots 0..y->rows-1 of a cache of capacity y->rows) into y
 * (Sec. 3.1 reconstruction with the Eq. 2 dequantization).
 */
int tac_decode(const void* codes, const void* norms, const tac_layer_cfg* cfg, tac_rows* y,
               tac_stream_t stream);

/*
 * Batched encode.  Jobs may mix d, input dtypes and codebooks; jobs that share
 * the kernel shape (d, dtype, n_angle, norm_bits, norm_mode) run in one launch
 * (one per TAC_MAX_JOBS such jobs).  With several launches they run
 * concurrently, largest first: the first on `stream`, the others on
 * library-owned streams that wait for `stream` at the call (an event), while
 * `stream` waits for them before the call returns (events), so the call's work
 * is ordered on `stream` as if it ran there alone and may be captured into a
 * CUDA graph.  A call with fewer than 640 warp tiles (4-row d = 128 tiles,
 * 8-row d = 64 tiles, ...) per SM in all gives each launch a share of the SMs
 * in proportion to its tiles, so that its launches run side by side; larger
 * calls give every launch the whole GPU.  Each launch is followed by its
 * fix-up kernel (see tac_encode_multi_ws): in a small call on the launch's
 * stream right after it, in a larger one after all of the call's encode
 * launches (a second fork / join), the fix-ups side by side.  The first call
 * with several launches on a device creates three streams and four events
 * (kept for the process); make it outside stream capture.  With `slot` the
 * rows of a decode step land at per-sequence record slots (streaming append).
 * Jobs must not write overlapping slots.
 */
int tac_encode_multi(const tac_encode_job* jobs, int njobs, tac_stream_t stream);

/*
 * The encode's re-decision workspace.  The fast path decides every code in
 * fp32 and certifies it against a bound on its own error (Alg. 1's edge test,
 * Eq. 2's rounding); each launch appends the codes it could not certify (a few
 * in ten thousand) to a queue in this workspace, and a fix-up kernel on the
 * launch's stream re-decides them (double-float, then exact integer sums).
 *
 * tac_encode_workspace_bytes returns the recommended size for the call
 * tac_encode_multi_ws(jobs, njobs, ...) (queue room for one code in 512 of
 * every group, far above the rates of the paper's workloads) and stores the
 * minimum in *min_bytes (if not NULL): per launch a counter block, one bit per
 * row and a copy of the launch's job table.
 * With less than the recommended size the queues shrink; a code that finds its
 * queue full has its whole row re-decided instead, so the results do not depend
 * on the size, only the time does.  Returns -1 (tac_last_error) for a call
 * tac_encode_multi would reject.
 *
 * tac_encode_multi_ws is tac_encode_multi with the caller's workspace (device
 * memory, 16-byte aligned, at least the minimum; its contents need no
 * initialization; it must not be used by other work until the call's work on
 * `stream` is done).  TAC_E_INVAL if the workspace is too small.
 */
int64_t tac_encode_workspace_bytes(const tac_encode_job* jobs, int njobs, int64_t* min_bytes);
int tac_encode_multi_ws(const tac_encode_job* jobs, int njobs, void* workspace, int64_t workspace_bytes,
                        tac_stream_t stream);

/* Batched decode, grouped into launches (run concurrently) like tac_encode_multi. */
int tac_decode_multi(const tac_decode_job* jobs, int njobs, tac_stream_t stream);

/*
 * Attention straight from the records (a consumer of the Sec. 3.1
 * reconstruction; the paper has no counterpart: it evaluates its codes through
 * a model's attention without a kernel for it).  For each of the job's nq
 * query rows q_a, over the record slots t = 0 .. tokens-1 of a K and a V cache:
 *   s_t = scale * (q_a . k^_t),   out_a = sum_t softmax(s)_t v^_t,
 * where k^_t, v^_t are the rows tac_decode would produce.  Because H and D are
 * orthogonal, s_t = scale * ((H D_K q_a) . y^K_t) and out_a = D_V H (sum_t p_t y^V_t)
 * with y^ = r^ (cos, sin)(2 pi k / n): no record is transformed back.
 * Results agree with decode-then-attend up to fp32 rounding (not bit-exact).
 */
#define TAC_MAX_QUERIES 8      /* query rows per job (a GQA group) */
#define TAC_ATTEND_MAX_JOBS 160 /* jobs per launch pair of tac_attend_multi */
#define TAC_ATTEND_SPLIT 256   /* tokens per partial result in the workspace */

typedef struct {
  tac_layer_cfg cfg_k;     /* K codebook and D; cfg_v.d must equal cfg_k.d (64 or 128) */
  tac_layer_cfg cfg_v;     /* V codebook and D */
  const void* k_codes;     /* K cache planes (device), capacity slots */
  const void* k_norms;
  const void* v_codes;     /* V cache planes (device), capacity slots */
  const void* v_norms;
  int64_t capacity;
  int64_t tokens;          /* 1 <= tokens <= capacity: attend to slots 0..tokens-1 */
  tac_rows q;              /* nq = q.rows query rows, 1 <= nq <= TAC_MAX_QUERIES (device) */
  tac_rows out;            /* nq output rows, same dtype as q (device) */
  float scale;             /* softmax scale, e.g. 1/sqrt(d) */
} tac_attend_job;

/* Device workspace bytes tac_attend_multi needs for these jobs:
 * sum over jobs of ceil(tokens / TAC_ATTEND_SPLIT) * nq * (d + 2) floats, each
 * job's part rounded up to 16 bytes.  Returns -1 for invalid jobs. */
int64_t tac_attend_workspace_bytes(const tac_attend_job* jobs, int njobs);

/* Attention for every job.  Jobs of one (d, dtype) share a launch pair (up to
 * TAC_ATTEND_MAX_JOBS jobs each); several launch pairs run concurrently on
 * `stream` and the helper streams of tac_encode_multi (fork / join by events),
 * ordered on `stream` as a whole.
 * `workspace` (device, 16-byte aligned, >= tac_attend_workspace_bytes) is the
 * caller's; its contents need no initialisation and are overwritten.  Calls
 * that share a workspace must not overlap in time. */
int tac_attend_multi(const tac_attend_job* jobs, int njobs, void* workspace, int64_t workspace_bytes,
                     tac_stream_t stream);

/*
 * tac_attend_multi without a caller workspace, for callers that cannot
 * allocate device memory (the paper has no counterpart: this is an interface
 * convenience of this library).  The partial results live in one static
 * device array of TAC_ATTEND_STATIC_WS_BYTES per device, built into the
 * library; nothing is allocated, on the device or the host heap.
 *
 *   - Same jobs, results and errors as tac_attend_multi with a workspace.
 *   - Jobs whose tac_attend_workspace_bytes exceeds TAC_ATTEND_STATIC_WS_BYTES
 *     are rejected with TAC_E_UNSUPPORTED (nothing launched); split them over
 *     several calls, or pass a workspace to tac_attend_multi.
 *   - Nothing in the array needs to start at zero: every partial record is
 *     written by the first kernel before the second reads it.
 *   - First call on each device: resolves the array's address with
 *     cudaGetSymbolAddress, which may load the library's attention module,
 *     and reads the device's SM count.  Make that first call outside stream
 *     capture; a call with njobs = 0 does only this setup and returns
 *     TAC_E_CUDA if it fails.  The address is cached per process and device;
 *     after cudaDeviceReset it is stale (the module is loaded anew), so such a
 *     process must not call this entry point again.  The first launch
 *     of each kernel shape (d, q dtype, query count) on a device also sets its
 *     shared-memory limit, as in tac_attend_multi.  After both, a call makes
 *     no CUDA runtime call but cudaGetDevice, the launches and
 *     cudaGetLastError, and can be captured into a CUDA graph.
 *   - All calls on one device share the array: two calls that overlap in time
 *     (different streams, or host threads without ordering) race on it and
 *     give undefined results.  Calls in one stream are ordered and safe.
 */
#define TAC_ATTEND_STATIC_WS_BYTES (8 << 20)
int tac_attend_multi_static(const tac_attend_job* jobs, int njobs, tac_stream_t stream);

/*
 * Transform only, for checking the butterfly: y = H D x (Sec. 2), normalized,
 * written as fp32 rows of d elements (row stride d).  signs: host words as in
 * tac_layer_cfg.signs.  d: any power of two 2..128.
 */
int tac_fwht_debug(const tac_rows* x, int d, const uint32_t* signs, float* y,
                   tac_stream_t stream);

/*
 * The hardware approximations the kernels use, element-wise, for tests that
 * measure them against the error bounds the encoder's certification assumes
 * (the paper has no counterpart).  op: 0 sqrt.approx.f32, 1 sqrt.approx.ftz.f32,
 * 2 rcp.approx.ftz.f32, 3 lg2.approx.f32, 4 lg2.approx.ftz.f32,
 * 5 ex2.approx.ftz.f32.  x, y: n floats (device, 16-byte aligned).
 */
int tac_hw_approx_debug(int op, const float* x, float* y, int64_t n, tac_stream_t stream);

/* Message of the last failed call on this host thread ("" if none). */
const char* tac_last_error(void);

/* Library version string. */
const char* tac_version(void);

#ifdef __cplusplus
}
#endif

#endif /* TAC_H_ */
