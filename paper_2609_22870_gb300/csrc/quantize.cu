// a1/a2: scaled E4M3 quantisation, S = max|X| / 448, codes = Q_FP8(X / S)
// (Eq. 3, §2.2) at tensor, row and block granularity.
//
// All kernels are HBM-bound streams over bf16 input: 128-bit loads of 8 bf16,
// block amax by warp shuffles, the correctly rounded float32 quotient x / S
// (__fdiv_rn), and the hardware float32 -> E4M3 conversion with round to
// nearest even and saturation to +-448 (__nv_cvt_float2_to_fp8x2,
// __NV_SATFINITE), stored as 64-bit groups of 8 codes.
#include <cuda_bf16.h>
#include <cuda_fp8.h>

#include "common.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

__device__ uint32_t d_status;

constexpr float kFmax = 448.0f;

__device__ __forceinline__ void unpack8(const uint4& v, float (&f)[8]) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 t = __bfloat1622float2(h[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}

__device__ __forceinline__ float amax8(const float (&f)[8], bool& finite) {
  float m = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    finite &= isfinite(f[i]);
    m = fmaxf(m, fabsf(f[i]));
  }
  return m;
}

// S = fl32(amax / 448), 1 when amax == 0.
__device__ __forceinline__ float scale_of(float amax) {
  return amax == 0.f ? 1.f : __fdiv_rn(amax, kFmax);
}

// Eight codes Q_FP8(fl32(x_i / S)), byte i = element i.
__device__ __forceinline__ uint2 encode8(const float (&f)[8], float s) {
  uint32_t w[2];
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    uint32_t acc = 0;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const float a = __fdiv_rn(f[4 * j + 2 * i], s);
      const float b = __fdiv_rn(f[4 * j + 2 * i + 1], s);
      const __nv_fp8x2_storage_t p =
          __nv_cvt_float2_to_fp8x2(make_float2(a, b), __NV_SATFINITE, __NV_E4M3);
      acc |= static_cast<uint32_t>(p) << (16 * i);
    }
    w[j] = acc;
  }
  return make_uint2(w[0], w[1]);
}

__device__ __forceinline__ void flag_bad() { atomicOr(&d_status, kErrDevice); }

// ---------------------------------------------------------------- tensor
// Global amax over the tensor (as float bits: |x| >= 0 orders like uint32).
__global__ void amax_kernel(const uint16_t* __restrict__ x, int64_t rows, int64_t cols, int64_t ld,
                            unsigned int* __restrict__ amax_bits) {
  const int64_t vpr = cols / 8;
  const int64_t nvec = rows * vpr;
  float m = 0.f;
  bool finite = true;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < nvec;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / vpr, c = (i - r * vpr) * 8;
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(x + r * ld + c));
    float f[8];
    unpack8(v, f);
    m = fmaxf(m, amax8(f, finite));
  }
  m = warp_max(m);
  if (!__all_sync(0xffffffffu, finite) && (threadIdx.x & 31) == 0) flag_bad();
  if ((threadIdx.x & 31) == 0) atomicMax(amax_bits, __float_as_uint(m));
}

__global__ void quant_tensor_kernel(const uint16_t* __restrict__ x, int64_t rows, int64_t cols,
                                    int64_t ld, uint8_t* __restrict__ codes,
                                    float* __restrict__ scales,
                                    const unsigned int* __restrict__ amax_bits) {
  const float s = scale_of(__uint_as_float(*amax_bits));
  if (blockIdx.x == 0 && threadIdx.x == 0) scales[0] = s;
  const int64_t vpr = cols / 8;
  const int64_t nvec = rows * vpr;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < nvec;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / vpr, c = (i - r * vpr) * 8;
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(x + r * ld + c));
    float f[8];
    unpack8(v, f);
    *reinterpret_cast<uint2*>(codes + r * cols + c) = encode8(f, s);
  }
}

// ---------------------------------------------------------------- row
// One CTA per row; up to kRowVec vectors of 8 per thread stay in registers
// between the amax and the encode pass, longer rows are re-read.
constexpr int kRowThreads = 256;
constexpr int kRowVec = 4;

__global__ void __launch_bounds__(kRowThreads) quant_row_kernel(
    const uint16_t* __restrict__ x, int64_t rows, int64_t cols, int64_t ld,
    uint8_t* __restrict__ codes, float* __restrict__ scales) {
  __shared__ float red[kRowThreads / 32];
  const int64_t r = blockIdx.x;
  const uint16_t* xr = x + r * ld;
  uint8_t* cr = codes + r * cols;
  const int nvec = static_cast<int>(cols / 8);
  uint4 buf[kRowVec];
  float m = 0.f;
  bool finite = true;
  const bool cached = nvec <= kRowThreads * kRowVec;
  if (cached) {
#pragma unroll
    for (int j = 0; j < kRowVec; ++j) {
      const int v = threadIdx.x + j * kRowThreads;
      if (v < nvec) {
        buf[j] = __ldg(reinterpret_cast<const uint4*>(xr + v * 8));
        float f[8];
        unpack8(buf[j], f);
        m = fmaxf(m, amax8(f, finite));
      }
    }
  } else {
    for (int v = threadIdx.x; v < nvec; v += kRowThreads) {
      float f[8];
      unpack8(__ldg(reinterpret_cast<const uint4*>(xr + v * 8)), f);
      m = fmaxf(m, amax8(f, finite));
    }
  }
  m = warp_max(m);
  if (!__all_sync(0xffffffffu, finite) && (threadIdx.x & 31) == 0) flag_bad();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x / 32] = m;
  __syncthreads();
  m = red[0];
#pragma unroll
  for (int w = 1; w < kRowThreads / 32; ++w) m = fmaxf(m, red[w]);
  const float s = scale_of(m);
  if (threadIdx.x == 0) scales[r] = s;
  if (cached) {
#pragma unroll
    for (int j = 0; j < kRowVec; ++j) {
      const int v = threadIdx.x + j * kRowThreads;
      if (v < nvec) {
        float f[8];
        unpack8(buf[j], f);
        *reinterpret_cast<uint2*>(cr + v * 8) = encode8(f, s);
      }
    }
  } else {
    for (int v = threadIdx.x; v < nvec; v += kRowThreads) {
      float f[8];
      unpack8(__ldg(reinterpret_cast<const uint4*>(xr + v * 8)), f);
      *reinterpret_cast<uint2*>(cr + v * 8) = encode8(f, s);
    }
  }
}

// ---------------------------------------------------------------- 1x128 blocks
// 16 lanes per block of 128 (8 elements each); each warp covers kActUnroll
// pairs of blocks per iteration so several 16-byte loads are in flight.
// Scales are stored block-column major: scales[kb * rows + r].
constexpr int kActUnroll = 4;

__global__ void __launch_bounds__(256) quant_act_block_kernel(
    const uint16_t* __restrict__ x, int64_t rows, int64_t cols, int64_t ld,
    uint8_t* __restrict__ codes, float* __restrict__ scales) {
  const int64_t nkb = cols / 128;
  const int64_t nblk = rows * nkb;
  const int lane = threadIdx.x & 31;
  const int sub = lane & 15;
  const int64_t warp_id = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t base = warp_id * 2 * kActUnroll; base < nblk; base += nwarps * 2 * kActUnroll) {
    uint4 v[kActUnroll];
    int64_t blk[kActUnroll];
#pragma unroll
    for (int u = 0; u < kActUnroll; ++u) {
      blk[u] = base + 2 * u + (lane >> 4);
      if (blk[u] < nblk) {
        const int64_t r = blk[u] / nkb, kb = blk[u] - r * nkb;
        v[u] = __ldg(reinterpret_cast<const uint4*>(x + r * ld + kb * 128 + sub * 8));
      } else {
        v[u] = make_uint4(0, 0, 0, 0);
      }
    }
#pragma unroll
    for (int u = 0; u < kActUnroll; ++u) {
      float f[8];
      unpack8(v[u], f);
      bool finite = true;
      float m = amax8(f, finite);
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      if (!finite) flag_bad();
      const float s = scale_of(m);
      if (blk[u] < nblk) {
        const int64_t r = blk[u] / nkb, kb = blk[u] - r * nkb;
        *reinterpret_cast<uint2*>(codes + r * cols + kb * 128 + sub * 8) = encode8(f, s);
        if (sub == 0) scales[kb * rows + r] = s;
      }
    }
  }
}

// ---------------------------------------------------------------- 128x128 blocks
// One CTA of 256 threads per weight block: thread t owns column group t % 16
// (8 columns) of rows t / 16 + 16 i, i < 8.  Tail rows beyond `rows` are
// skipped.  Scales: scales[rb * nkb + kb].
__global__ void __launch_bounds__(256) quant_weight_block_kernel(
    const uint16_t* __restrict__ x, int64_t rows, int64_t cols, int64_t ld,
    uint8_t* __restrict__ codes, float* __restrict__ scales) {
  __shared__ float red[8];
  const int64_t nkb = cols / 128;
  const int64_t rb = blockIdx.x / nkb, kb = blockIdx.x - rb * nkb;
  const int cg = threadIdx.x & 15, rs = threadIdx.x >> 4;
  uint4 v[8];
  float m = 0.f;
  bool finite = true;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t r = rb * 128 + rs + 16 * i;
    if (r < rows) {
      v[i] = __ldg(reinterpret_cast<const uint4*>(x + r * ld + kb * 128 + cg * 8));
      float f[8];
      unpack8(v[i], f);
      m = fmaxf(m, amax8(f, finite));
    }
  }
  m = warp_max(m);
  if (!__all_sync(0xffffffffu, finite) && (threadIdx.x & 31) == 0) flag_bad();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  m = red[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) m = fmaxf(m, red[w]);
  const float s = scale_of(m);
  if (threadIdx.x == 0) scales[rb * nkb + kb] = s;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t r = rb * 128 + rs + 16 * i;
    if (r < rows) {
      float f[8];
      unpack8(v[i], f);
      *reinterpret_cast<uint2*>(codes + r * cols + kb * 128 + cg * 8) = encode8(f, s);
    }
  }
}

int grid_for(int64_t work_items, int threads) {
  const int64_t want = (work_items + threads - 1) / threads;
  const int64_t cap = static_cast<int64_t>(sm_count()) * 8;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

}  // namespace

cudaError_t launch_quantize(const void* x, int64_t rows, int64_t cols, int64_t ld, int gran,
                            int role, uint8_t* codes, float* scales, void* ws, cudaStream_t s) {
  const uint16_t* xb = static_cast<const uint16_t*>(x);
  if (rows == 0) return cudaSuccess;
  if (gran == FP8RL_GRAN_TENSOR) {
    unsigned int* amax = static_cast<unsigned int*>(ws);
    cudaError_t e = cudaMemsetAsync(amax, 0, sizeof(unsigned int), s);
    if (e != cudaSuccess) return e;
    const int64_t nvec = rows * (cols / 8);
    amax_kernel<<<grid_for(nvec, 256), 256, 0, s>>>(xb, rows, cols, ld, amax);
    quant_tensor_kernel<<<grid_for(nvec, 256), 256, 0, s>>>(xb, rows, cols, ld, codes, scales,
                                                             amax);
  } else if (gran == FP8RL_GRAN_ROWWISE) {
    quant_row_kernel<<<static_cast<unsigned>(rows), kRowThreads, 0, s>>>(xb, rows, cols, ld,
                                                                          codes, scales);
  } else if (role == FP8RL_ROLE_ACT) {
    const int64_t nblk = rows * (cols / 128);
    quant_act_block_kernel<<<grid_for(nblk * 16, 256), 256, 0, s>>>(xb, rows, cols, ld, codes,
                                                                      scales);
  } else {
    const int64_t nrb = (rows + 127) / 128;
    quant_weight_block_kernel<<<static_cast<unsigned>(nrb * (cols / 128)), 256, 0, s>>>(
        xb, rows, cols, ld, codes, scales);
  }
  return cudaGetLastError();
}

uint32_t quantize_status_take() {
  uint32_t v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, d_status, sizeof(v)) != cudaSuccess) return 0;
  cudaMemcpyToSymbol(d_status, &z, sizeof(z));
  return v;
}

}  // namespace fp8rl
