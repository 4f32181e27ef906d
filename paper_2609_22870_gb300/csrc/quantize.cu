// a1/a2: scaled E4M3 quantisation, S = max|X| / 448, codes = Q_FP8(X / S)
// (Eq. 3, §2.2) at tensor, row and block granularity.
//
// All kernels are HBM-bound streams over bf16 input, so the work per element
// is kept to a few instructions (e4m3_encode.cuh): the block maximum of |x|
// on packed bf16 pairs, the correctly rounded quotient x / S by Markstein's
// correction on packed float pairs, and the hardware float32 -> E4M3
// conversion (round to nearest even, saturation to +-448), stored as 8-byte
// groups.
//
// Block granularities run a persistent kernel: a producer warp streams tiles
// of R rows x 128 columns into a ring of shared-memory stages by TMA, several
// tiles ahead, and eight consumer warps reduce and encode from shared memory.
// Row and tensor granularities read 16-byte groups straight from HBM.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "e4m3_encode.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

__device__ uint32_t d_status;

__device__ __forceinline__ void flag_bad() { atomicOr(&d_status, kErrDevice); }

// Float bits of the largest |x| in a packed running maximum (non-negative, so
// the bits order like the values; +inf and NaN sort above every finite value).
__device__ __forceinline__ uint32_t amax_bits(uint32_t m) { return __float_as_uint(amax_of(m)); }

constexpr uint32_t kInfBits = 0x7F800000u;

// Barrier `id` over the first `n` threads; returns the AND of `p` over them.
__device__ __forceinline__ bool bar_and(uint32_t id, uint32_t n, bool p) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "barrier.red.and.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(p)), "r"(id), "r"(n)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ void bar_sync(uint32_t id, uint32_t n) {
  asm volatile("barrier.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

// ---------------------------------------------------------------- tensor
// The per-tensor kernels walk the tensor as vectors of 8 bf16 (16 bytes):
// vector i sits at row i / vpr, column (i % vpr) * 8.  A contiguous tensor
// (ld == cols) is one linear array, read without that division; otherwise
// each thread carries its (row, column) and steps it by the grid stride.
// Four vectors per thread and step keep 64 bytes in flight per thread.
struct VecWalk {
  const uint16_t* x;
  int64_t vpr, ld;
  __device__ __forceinline__ int64_t offset(int64_t i) const {
    if (ld == vpr * 8) return i * 8;
    const int64_t r = i / vpr;
    return r * ld + (i - r * vpr) * 8;
  }
};

// Global amax over the tensor, as float bits (atomicMax on the bits).
__global__ void amax_kernel(const uint16_t* __restrict__ x, int64_t rows, int64_t cols, int64_t ld,
                            unsigned int* __restrict__ amax) {
  const VecWalk vw{x, cols / 8, ld};
  const int64_t nvec = rows * vw.vpr;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  uint32_t m = 0;
  int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  for (; i + 3 * stride < nvec; i += 4 * stride) {
    uint4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) v[u] = __ldg(reinterpret_cast<const uint4*>(x + vw.offset(i + u * stride)));
#pragma unroll
    for (int u = 0; u < 4; ++u) m = amax_bf16x8(m, v[u]);
  }
  for (; i < nvec; i += stride) m = amax_bf16x8(m, __ldg(reinterpret_cast<const uint4*>(x + vw.offset(i))));
  const uint32_t b = __reduce_max_sync(0xffffffffu, amax_bits(m));
  if ((threadIdx.x & 31) == 0) {
    if (b >= kInfBits) flag_bad();
    atomicMax(amax, b);
  }
}

__global__ void quant_tensor_kernel(const uint16_t* __restrict__ x, int64_t rows, int64_t cols,
                                    int64_t ld, uint8_t* __restrict__ codes,
                                    float* __restrict__ scales,
                                    const unsigned int* __restrict__ amax, bool pow2) {
  const float s = e4m3_scale(__uint_as_float(*amax), pow2);
  const E4M3Enc e = e4m3_encoder(s);
  if (blockIdx.x == 0 && threadIdx.x == 0) scales[0] = s;
  const VecWalk vw{x, cols / 8, ld};
  const int64_t nvec = rows * vw.vpr;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  // codes are [rows][cols] contiguous: vector i's codes start at byte i * 8
  for (; i + 3 * stride < nvec; i += 4 * stride) {
    uint4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) v[u] = __ldg(reinterpret_cast<const uint4*>(x + vw.offset(i + u * stride)));
#pragma unroll
    for (int u = 0; u < 4; ++u) *reinterpret_cast<uint2*>(codes + (i + u * stride) * 8) = e4m3_encode8(v[u], e);
  }
  for (; i < nvec; i += stride)
    *reinterpret_cast<uint2*>(codes + i * 8) = e4m3_encode8(__ldg(reinterpret_cast<const uint4*>(x + vw.offset(i))), e);
}

// ---------------------------------------------------------------- row
// One CTA per row; up to kRowVec 16-byte groups per thread stay in registers
// between the amax and the encode pass, longer rows are re-read.
constexpr int kRowThreads = 256;
constexpr int kRowVec = 4;

__global__ void __launch_bounds__(kRowThreads) quant_row_kernel(
    const uint16_t* __restrict__ x, int64_t rows, int64_t cols, int64_t ld,
    uint8_t* __restrict__ codes, float* __restrict__ scales, bool pow2) {
  __shared__ uint32_t red[kRowThreads / 32];
  const int64_t r = blockIdx.x;
  const uint16_t* xr = x + r * ld;
  uint8_t* cr = codes + r * cols;
  const int nvec = static_cast<int>(cols / 8);
  uint4 buf[kRowVec];
  uint32_t m = 0;
  const bool cached = nvec <= kRowThreads * kRowVec;
  if (cached) {
#pragma unroll
    for (int j = 0; j < kRowVec; ++j) {
      const int v = threadIdx.x + j * kRowThreads;
      if (v < nvec) {
        buf[j] = __ldg(reinterpret_cast<const uint4*>(xr + v * 8));
        m = amax_bf16x8(m, buf[j]);
      }
    }
  } else {
    for (int v = threadIdx.x; v < nvec; v += kRowThreads)
      m = amax_bf16x8(m, __ldg(reinterpret_cast<const uint4*>(xr + v * 8)));
  }
  const uint32_t wb = __reduce_max_sync(0xffffffffu, amax_bits(m));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x / 32] = wb;
  __syncthreads();
  uint32_t b = red[0];
#pragma unroll
  for (int w = 1; w < kRowThreads / 32; ++w) b = max(b, red[w]);
  if (threadIdx.x == 0 && b >= kInfBits) flag_bad();
  const float s = e4m3_scale(__uint_as_float(b), pow2);
  const E4M3Enc e = e4m3_encoder(s);
  if (threadIdx.x == 0) scales[r] = s;
  if (cached) {
#pragma unroll
    for (int j = 0; j < kRowVec; ++j) {
      const int v = threadIdx.x + j * kRowThreads;
      if (v < nvec) *reinterpret_cast<uint2*>(cr + v * 8) = e4m3_encode8(buf[j], e);
    }
  } else {
    for (int v = threadIdx.x; v < nvec; v += kRowThreads)
      *reinterpret_cast<uint2*>(cr + v * 8) =
          e4m3_encode8(__ldg(reinterpret_cast<const uint4*>(xr + v * 8)), e);
  }
}

// ---------------------------------------------------------------- streamed blocks
// Persistent CTAs of 8 consumer warps + 1 producer warp walk the tiles of
// R rows x 128 columns (R = 32: 32 rows of 1x128 activation blocks; R = 128:
// one 128x128 weight block), tile t = rb * (cols / 128) + kb, CTA b taking
// t = b, b + grid, ...  The producer's elected lane issues a TMA 2-D load per
// tile (rows of 256 bytes, no swizzle, rows past the matrix read as zeros)
// into stage j % kStages and waits for that stage's `empty` barrier (one
// arrival per consumer warp) before reusing it; consumers wait for `full`,
// copy their part of the tile into registers, release the stage and encode.
// Activation scales: scales[kb * rows + r]; weight scales:
// scales[rb * (cols / 128) + kb].  Every wait is bounded by `limit_ns`: on
// expiry the CTA raises the timeout status, stops, and the producer waits
// (bounded again) for its copies still in flight before the CTA exits.
template <int R>
struct Stream {
  static constexpr int kStages = (R == 128) ? 3 : 8;
  static constexpr int kCtasPerSm = (R == 128) ? 2 : 3;
  static constexpr uint32_t kTileBytes = R * 256;
  static constexpr int kThreads = 288;
  static constexpr size_t kSmem = kStages * kTileBytes + 1024 + 2 * 8 * kStages;
};

template <int R, bool POW2>
__global__ void __launch_bounds__(288) quant_block_stream_kernel(
    const __grid_constant__ CUtensorMap tmx, int64_t rows, int64_t cols,
    uint8_t* __restrict__ codes, float* __restrict__ scales, uint64_t limit_ns) {
  constexpr int S = Stream<R>::kStages;
  constexpr uint32_t TB = Stream<R>::kTileBytes;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * TB);
  uint64_t* empty = full + S;
  __shared__ uint32_t red[8];
  __shared__ int abort_s;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t nkb = cols / 128;
  const int64_t ntiles = (rows + R - 1) / R * nkb;
  if (tid == 0) {
    for (int j = 0; j < S; ++j) {
      mbar_init(smem_u32(&full[j]), 1);
      mbar_init(smem_u32(&empty[j]), 8);
    }
    abort_s = 0;
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == 8) {  // ------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tmx);
      int j = 0;
      for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x, ++j) {
        const int stage = j % S;
        if (j >= S && !mbar_wait(smem_u32(&empty[stage]), ((j / S) + 1) & 1, limit_ns, &abort_s)) {
          abort_s = 1;
          atomicOr(&d_status, kErrTimeout);
          break;
        }
        const int64_t rb = t / nkb, kb = t - rb * nkb;
        mbar_arrive_expect_tx(smem_u32(&full[stage]), TB);
        tma_load_2d(smem_u32(smem + stage * TB), &tmx, smem_u32(&full[stage]),
                    static_cast<int32_t>(kb * 128), static_cast<int32_t>(rb * R));
      }
      // no copy may still be landing when the CTA exits: wait for the last
      // copy of every stage (its phase is the stage's latest)
      for (int k = (j > S ? j - S : 0); k < j; ++k)
        if (!mbar_wait(smem_u32(&full[k % S]), (k / S) & 1, limit_ns, nullptr))
          atomicOr(&d_status, kErrTimeout);
    }
    return;
  }

  // ------------------------------------------------------------ consumers
  bool finite = true, ok = true;
  int j = 0;
  for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x, ++j) {
    const int stage = j % S;
    const uint8_t* tile = smem + stage * TB;
    const int64_t rb = t / nkb, kb = t - rb * nkb;
    if (R == 32) {
      // warp w owns tile rows 4w .. 4w+3; 8 lanes per row, 16 bf16 per lane
      ok = __all_sync(0xffffffffu,
                      mbar_wait(smem_u32(&full[stage]), (j / S) & 1, limit_ns, &abort_s));
      if (!ok) break;
      const int rr = warp * 4 + (lane >> 3), c = lane & 7;
      const uint4 v0 = *reinterpret_cast<const uint4*>(tile + rr * 256 + c * 16);
      const uint4 v1 = *reinterpret_cast<const uint4*>(tile + rr * 256 + c * 16 + 128);
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&empty[stage]));
      uint32_t b = amax_bits(amax_bf16x8(amax_bf16x8(0u, v0), v1));
      b = max(b, __shfl_xor_sync(0xffffffffu, b, 4));
      b = max(b, __shfl_xor_sync(0xffffffffu, b, 2));
      b = max(b, __shfl_xor_sync(0xffffffffu, b, 1));
      finite &= b < kInfBits;
      const float s = e4m3_scale(__uint_as_float(b), POW2);
      const E4M3Enc e = e4m3_encoder(s);
      const uint2 c0 = e4m3_encode8(v0, e), c1 = e4m3_encode8(v1, e);
      const int64_t r = rb * R + rr;
      if (r < rows) {
        uint8_t* dst = codes + r * cols + kb * 128 + c * 8;
        *reinterpret_cast<uint2*>(dst) = c0;
        *reinterpret_cast<uint2*>(dst + 64) = c1;
        if (c == 0) scales[kb * rows + r] = s;
      }
    } else {
      // one block per tile: thread t owns 16-byte column group t % 16 of
      // rows t / 16 + 16 i
      ok = bar_and(1, 256, mbar_wait(smem_u32(&full[stage]), (j / S) & 1, limit_ns, &abort_s));
      if (!ok) break;
      const int cg = tid & 15, rsub = tid >> 4;
      uint4 v[8];
      uint32_t m = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        v[i] = *reinterpret_cast<const uint4*>(tile + (rsub + 16 * i) * 256 + cg * 16);
        m = amax_bf16x8(m, v[i]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&empty[stage]));
      const uint32_t wb = __reduce_max_sync(0xffffffffu, amax_bits(m));
      if (lane == 0) red[warp] = wb;
      bar_sync(2, 256);
      uint32_t b = red[0];
#pragma unroll
      for (int w = 1; w < 8; ++w) b = max(b, red[w]);
      finite &= b < kInfBits;
      const float s = e4m3_scale(__uint_as_float(b), POW2);
      const E4M3Enc e = e4m3_encoder(s);
      if (tid == 0) scales[rb * nkb + kb] = s;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int64_t r = rb * R + rsub + 16 * i;
        if (r < rows)
          *reinterpret_cast<uint2*>(codes + r * cols + kb * 128 + cg * 8) = e4m3_encode8(v[i], e);
      }
    }
  }
  if (!ok && lane == 0) {
    abort_s = 1;
    atomicOr(&d_status, kErrTimeout);
  }
  if (!__all_sync(0xffffffffu, finite) && lane == 0) flag_bad();
}

bool make_bf16_tmap(CUtensorMap* tm, const void* x, int64_t rows, int64_t cols, int64_t ld,
                    uint32_t box_rows) {
  auto fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(tensormap_encoder());
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {128, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int R, bool POW2>
cudaError_t launch_stream(const void* x, int64_t rows, int64_t cols, int64_t ld, uint8_t* codes,
                          float* scales, cudaStream_t s) {
  CUtensorMap tm;
  if (!make_bf16_tmap(&tm, x, rows, cols, ld, R)) return cudaErrorInvalidValue;
  auto kern = quant_block_stream_kernel<R, POW2>;
  static int configured_device = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured_device != dev) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(Stream<R>::kSmem));
    if (e != cudaSuccess) return e;
    configured_device = dev;
  }
  const int64_t ntiles = (rows + R - 1) / R * (cols / 128);
  const int64_t cap = static_cast<int64_t>(sm_count()) * Stream<R>::kCtasPerSm;
  const int grid = static_cast<int>(ntiles < cap ? ntiles : cap);
  kern<<<grid, Stream<R>::kThreads, Stream<R>::kSmem, s>>>(tm, rows, cols, codes, scales,
                                                           wait_limit_ns());
  return cudaGetLastError();
}

int grid_for(int64_t work_items, int threads) {
  const int64_t want = (work_items + threads - 1) / threads;
  const int64_t cap = static_cast<int64_t>(sm_count()) * 8;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

}  // namespace

cudaError_t launch_quantize(const void* x, int64_t rows, int64_t cols, int64_t ld, int gran,
                            int role, uint8_t* codes, float* scales, void* ws, bool pow2,
                            cudaStream_t s) {
  const uint16_t* xb = static_cast<const uint16_t*>(x);
  if (rows == 0) return cudaSuccess;
  if (gran == FP8RL_GRAN_TENSOR) {
    unsigned int* amax = static_cast<unsigned int*>(ws);
    cudaError_t e = cudaMemsetAsync(amax, 0, sizeof(unsigned int), s);
    if (e != cudaSuccess) return e;
    const int64_t nvec = rows * (cols / 8);
    amax_kernel<<<grid_for(nvec, 256), 256, 0, s>>>(xb, rows, cols, ld, amax);
    quant_tensor_kernel<<<grid_for(nvec, 256), 256, 0, s>>>(xb, rows, cols, ld, codes, scales,
                                                             amax, pow2);
  } else if (gran == FP8RL_GRAN_ROWWISE) {
    quant_row_kernel<<<static_cast<unsigned>(rows), kRowThreads, 0, s>>>(xb, rows, cols, ld,
                                                                          codes, scales, pow2);
  } else if (role == FP8RL_ROLE_ACT) {
    return pow2 ? launch_stream<32, true>(x, rows, cols, ld, codes, scales, s)
                : launch_stream<32, false>(x, rows, cols, ld, codes, scales, s);
  } else {
    return pow2 ? launch_stream<128, true>(x, rows, cols, ld, codes, scales, s)
                : launch_stream<128, false>(x, rows, cols, ld, codes, scales, s);
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
