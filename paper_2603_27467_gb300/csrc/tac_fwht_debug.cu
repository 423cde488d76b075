// Transform-only kernel y = H D x (Sec. 2: random +-1 diagonal, then the
// normalized Walsh-Hadamard butterfly), fp32 out.  It exists so the butterfly
// can be checked against a dense Hadamard matrix element by element; the
// encode/decode kernels use the same in-register butterfly.
#include "tac_common.cuh"

namespace tac {

struct FwhtParams {
  const void* x;
  float* y;
  int64_t rows;
  int64_t stride;  // elements
  int32_t dtype;
  uint32_t signs[4];
};

template <int D>
__global__ void __launch_bounds__(128) fwht_debug_kernel(const __grid_constant__ FwhtParams p) {
  const int64_t row = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (row >= p.rows) return;
  float v[D];
#pragma unroll
  for (int j = 0; j < D; ++j) {
    float x;
    if (p.dtype == TAC_BF16) {
      const uint16_t b = reinterpret_cast<const uint16_t*>(p.x)[row * p.stride + j];
      x = __uint_as_float((uint32_t)b << 16);
    } else {
      x = reinterpret_cast<const float*>(p.x)[row * p.stride + j];
    }
    v[j] = ((p.signs[j >> 5] >> (j & 31)) & 1u) ? -x : x;
  }
#pragma unroll
  for (int h = 1; h < D; h <<= 1) {
#pragma unroll
    for (int j = 0; j < D; ++j) {
      if ((j & h) == 0) {
        const float a = v[j], b = v[j + h];
        v[j] = __fadd_rn(a, b);
        v[j + h] = __fsub_rn(a, b);
      }
    }
  }
  // 1/sqrt(d): a power of two (exact) for d = 4^m, else 1/sqrt(d) rounded twice.
  float norm;
  if (D == 4) norm = 0.5f;
  else if (D == 16) norm = 0.25f;
  else if (D == 64) norm = 0.125f;
  else norm = __fdiv_rn(1.0f, __fsqrt_rn((float)D));
#pragma unroll
  for (int j = 0; j < D; ++j) p.y[row * D + j] = __fmul_rn(v[j], norm);
}

cudaError_t launch_fwht_debug(int d, const void* x, int dtype, int64_t rows, int64_t stride,
                              const uint32_t* signs, float* y, cudaStream_t st) {
  FwhtParams p;
  p.x = x; p.y = y; p.rows = rows; p.stride = stride; p.dtype = dtype;
  for (int q = 0; q < 4; ++q) p.signs[q] = (q < (d + 31) / 32) ? signs[q] : 0u;
  if (rows == 0) return cudaSuccess;
  const int threads = 128;
  const unsigned grid = (unsigned)((rows + threads - 1) / threads);
  switch (d) {
    case 2: fwht_debug_kernel<2><<<grid, threads, 0, st>>>(p); break;
    case 4: fwht_debug_kernel<4><<<grid, threads, 0, st>>>(p); break;
    case 8: fwht_debug_kernel<8><<<grid, threads, 0, st>>>(p); break;
    case 16: fwht_debug_kernel<16><<<grid, threads, 0, st>>>(p); break;
    case 32: fwht_debug_kernel<32><<<grid, threads, 0, st>>>(p); break;
    case 64: fwht_debug_kernel<64><<<grid, threads, 0, st>>>(p); break;
    case 128: fwht_debug_kernel<128><<<grid, threads, 0, st>>>(p); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

// Element-wise hardware approximations, as the kernels use them (tac_common.cuh):
// op 0 sqrt.approx.f32, 1 sqrt.approx.ftz.f32, 2 rcp.approx.ftz.f32,
// 3 lg2.approx.f32, 4 lg2.approx.ftz.f32, 5 ex2.approx.ftz.f32.
__global__ void __launch_bounds__(256) hw_approx_kernel(int op, const float* __restrict__ x, float* __restrict__ y,
                                                        int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const float a = x[i];
    float r;
    switch (op) {
      case 0: r = sqrt_approx(a); break;
      case 1: r = sqrt_ftz(a); break;
      case 2: r = rcp_approx(a); break;
      case 3: r = lg2_approx(a); break;
      case 4: r = lg2_ftz(a); break;
      default: r = ex2_ftz(a); break;
    }
    y[i] = r;
  }
}

cudaError_t launch_hw_approx(int op, const float* x, float* y, int64_t n, int sms, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  int64_t blocks = (n + 255) / 256;
  const int64_t cap = (int64_t)(sms > 0 ? sms : 1) * 8;
  if (blocks > cap) blocks = cap;
  hw_approx_kernel<<<(unsigned)blocks, 256, 0, st>>>(op, x, y, n);
  return cudaGetLastError();
}

}  // namespace tac
