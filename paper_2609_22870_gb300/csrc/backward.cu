// Backward through the FP8 lm_head with FP8 contractions.  Given
// g_t = dLoss/dlogp_t (the clipped surrogate's gradient) and the forward
// pass's lse, the chain rule through the log-softmax gives
// P[t][v] = dLoss/dz[t][v] = g_t (1{v == y_t} - exp(z[t][v] - lse_t)), and
// through z = h W^T the two contractions
//   dh = P W  ([T][V] x [V][H], K = V),     dW = P^T h  ([V][T] x [T][H], K = T).
// The quantisers pass the gradient straight through; every operand of the two
// contractions is E4M3-quantised along its own K axis (the paper trains with
// FP8 GEMMs in the backward pass as well, §3 and the performance appendix):
//   1. the FP8 GEMM recomputes z tile by tile and its epilogue writes the
//      codes of P with 1x128 scales along V and the codes of P^T with
//      128 x 128 scales (the float32 logits and P are never stored);
//   2. W [V][H] and h [T][H] (bf16) are transposed and quantised to W^T
//      [H][V'] and h^T [H][T'] with 128 x 128 scales (V', T' = V, T rounded
//      up to 128; the padding holds zero codes);
//   3. the block-scaled FP8 GEMM forms dh and dW into float32.
// With pow2_scales (implied by power-of-two forward scales, the UE8M0
// variant) P, P^T, W^T and h^T take power-of-two scales (floored at 2^-127)
// and both contractions run on the block-scaled MMA (tcgen05.mma
// kind::mxf8f6f4), which applies them per 32-wide K step; the recompute runs
// in the forward's own mode.
#include <cuda_fp8.h>

#include <algorithm>

#include "common.cuh"
#include "e4m3_encode.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

__device__ uint32_t d_status;

constexpr int kQT = 128;  // edge of a quantisation block / transpose tile

// codes[c][r] = Q_FP8(in[r][c] / S) for one 128 x 128 tile of the bf16 matrix
// in[rows][cols]: S = fl32(amax / 448) over the tile (1 when it is all zero;
// with pow2 the power of two above it, floored at 2^-127), written to
// scales[c / 128][r / 128] (row stride ld_out / 128).  The tile goes
// through shared memory (row pitch 136 bf16, so column reads by a warp hit
// distinct banks); each thread encodes 64 codes of one output row.  Rows of
// `in` past `rows` read as zero, so the padding columns of the codes are zero.
__global__ void __launch_bounds__(256) transpose_quantize_kernel(const uint16_t* __restrict__ in, int64_t rows,
                                                                 int64_t cols, int64_t ld_in,
                                                                 uint8_t* __restrict__ codes,
                                                                 float* __restrict__ scales, int64_t ld_out,
                                                                 int pow2) {
  constexpr int kPitch = kQT + 8;
  __shared__ __align__(16) uint16_t tile[kQT][kPitch];
  __shared__ uint32_t warp_max[8];
  const int64_t r0 = static_cast<int64_t>(blockIdx.x) * kQT;
  const int64_t c0 = static_cast<int64_t>(blockIdx.y) * kQT;
  const int tid = threadIdx.x;
  uint32_t m = 0;  // running max of |x| as packed bf16x2 (NaN-propagating)
  // 128 rows x 16 groups of 8 bf16; cols % 8 == 0 and ld_in % 8 == 0, so a
  // group is either wholly inside the matrix or wholly outside
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int idx = tid + k * 256;
    const int r = idx >> 4, gq = idx & 15;
    const int64_t gr = r0 + r, gc = c0 + gq * 8;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (gr < rows && gc < cols) v = __ldg(reinterpret_cast<const uint4*>(in + gr * ld_in + gc));
    *reinterpret_cast<uint4*>(&tile[r][gq * 8]) = v;
    m = amax_bf16x8(m, v);
  }
  const float a = amax_of(m);
  if (!(a <= 3.4e38f)) atomicOr(&d_status, kErrDevice);  // inf or NaN input
  const uint32_t wm = __reduce_max_sync(0xffffffffu, __float_as_uint(a));
  if ((tid & 31) == 0) warp_max[tid >> 5] = wm;
  __syncthreads();
  uint32_t bm = warp_max[0];
#pragma unroll
  for (int i = 1; i < 8; ++i) bm = max(bm, warp_max[i]);
  const float s = pow2 ? e8m0_floor(e4m3_scale(__uint_as_float(bm), true)) : e4m3_scale(__uint_as_float(bm), false);
  const E4M3Enc e = e4m3_encoder(s);
  // output row c = tid / 2 (column c of the tile), codes r = 64 (tid % 2) ..
  const int c = tid >> 1, rh = (tid & 1) * 64;
  if (c0 + c < cols) {
    uint4* dst = reinterpret_cast<uint4*>(codes + (c0 + c) * ld_out + r0 + rh);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint2 w[2];
#pragma unroll
      for (int h8 = 0; h8 < 2; ++h8) {
        const int rb = rh + q * 16 + h8 * 8;
        uint4 v;
        v.x = tile[rb + 0][c] | (static_cast<uint32_t>(tile[rb + 1][c]) << 16);
        v.y = tile[rb + 2][c] | (static_cast<uint32_t>(tile[rb + 3][c]) << 16);
        v.z = tile[rb + 4][c] | (static_cast<uint32_t>(tile[rb + 5][c]) << 16);
        v.w = tile[rb + 6][c] | (static_cast<uint32_t>(tile[rb + 7][c]) << 16);
        w[h8] = e4m3_encode8(v, e);
      }
      dst[q] = make_uint4(w[0].x, w[0].y, w[1].x, w[1].y);
    }
  }
  if (tid == 0) scales[(c0 / kQT) * (ld_out / kQT) + r0 / kQT] = s;
}

}  // namespace

BwdLayout bwd_layout(int64_t T, int64_t H, int64_t V) {
  BwdLayout l;
  l.vp = (V + kQT - 1) / kQT * kQT;
  l.tp = (T + kQT - 1) / kQT * kQT;
  const int64_t hb = (H + kQT - 1) / kQT;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes, 256);
    return at;
  };
  l.p = take(static_cast<size_t>(T) * l.vp);
  l.ps = take(static_cast<size_t>(l.vp / kQT) * T * 4);
  l.pt = take(static_cast<size_t>(V) * l.tp);
  l.pts = take(static_cast<size_t>(l.tp / kQT) * V * 4);
  l.wt = take(static_cast<size_t>(H) * l.vp);
  l.wts = take(static_cast<size_t>(hb) * (l.vp / kQT) * 4);
  l.ht = take(static_cast<size_t>(H) * l.tp);
  l.hts = take(static_cast<size_t>(hb) * (l.tp / kQT) * 4);
  // UE8M0 variant: scale images of the recompute, then of dh, then of dW
  // (one buffer: the three GEMMs run in stream order)
  l.sf = take(std::max({gemm_ue8m0_image_bytes(T, V, H), gemm_ue8m0_image_bytes(T, H, l.vp),
                        gemm_ue8m0_image_bytes(V, H, l.tp)}));
  l.total = off;
  return l;
}

cudaError_t launch_lm_head_backward(const uint8_t* hc, const float* hs, const uint8_t* wc,
                                    const float* wsc, int gran, int64_t T, int64_t H, int64_t V,
                                    const int32_t* targets, const float* lse, const float* grad,
                                    const uint16_t* h, const uint16_t* W, float* dh, float* dW,
                                    bool accumulate_dw, bool pow2_scales, void* ws, cudaStream_t s) {
  const BwdLayout l = bwd_layout(T, H, V);
  char* base = static_cast<char*>(ws);
  uint8_t* Pq = reinterpret_cast<uint8_t*>(base + l.p);
  float* Ps = reinterpret_cast<float*>(base + l.ps);
  uint8_t* Ptq = reinterpret_cast<uint8_t*>(base + l.pt);
  float* Pts = reinterpret_cast<float*>(base + l.pts);
  uint8_t* Wtq = reinterpret_cast<uint8_t*>(base + l.wt);
  float* Wts = reinterpret_cast<float*>(base + l.wts);
  uint8_t* Htq = reinterpret_cast<uint8_t*>(base + l.ht);
  float* Hts = reinterpret_cast<float*>(base + l.hts);
  const bool ue = pow2_scales || gran == FP8RL_GRAN_BLOCK_UE8M0;
  const int bgran = ue ? FP8RL_GRAN_BLOCK_UE8M0 : FP8RL_GRAN_BLOCK;
  uint8_t* sf = reinterpret_cast<uint8_t*>(base + l.sf);
  // 1. recompute z (FP8), quantise P = dLoss/dz in both orientations
  GemmArgs a{};
  a.a_codes = hc;
  a.a_scales = hs;
  a.b_codes = wc;
  a.b_scales = wsc;
  a.gran = gran;
  a.M = T;
  a.N = V;
  a.K = H;
  a.targets = targets;
  a.lse = lse;
  a.grad = grad;
  a.pq_out = Pq;
  a.pq_scales = Ps;
  a.ptq_out = Ptq;
  a.ptq_scales = Pts;
  a.ld_pq = l.vp;
  a.ld_ptq = l.tp;
  a.sf_images = sf;
  a.p_pow2 = ue ? 1 : 0;
  cudaError_t e = launch_gemm_dense_dlogits(a, s);
  if (e != cudaSuccess) return e;
  if (dh) {  // 2./3. dh[T][H] = P[T][V'] . (W^T[H][V'])^T
    e = launch_transpose_quantize(W, V, H, H, Wtq, Wts, l.vp, ue, s);
    if (e != cudaSuccess) return e;
    GemmArgs d{};
    d.a_codes = Pq;
    d.a_scales = Ps;
    d.b_codes = Wtq;
    d.b_scales = Wts;
    d.gran = bgran;
    d.sf_images = sf;
    d.M = T;
    d.N = H;
    d.K = l.vp;
    d.lda = l.vp;
    d.ldb = l.vp;
    d.c_out = dh;
    d.ld_c = H;
    e = launch_gemm_store(d, s);
    if (e != cudaSuccess) return e;
  }
  if (dW) {  // dW[V][H] = P^T[V][T'] . (h^T[H][T'])^T
    e = launch_transpose_quantize(h, T, H, H, Htq, Hts, l.tp, ue, s);
    if (e != cudaSuccess) return e;
    GemmArgs d{};
    d.a_codes = Ptq;
    d.a_scales = Pts;
    d.b_codes = Htq;
    d.b_scales = Hts;
    d.gran = bgran;
    d.sf_images = sf;
    d.M = V;
    d.N = H;
    d.K = l.tp;
    d.lda = l.tp;
    d.ldb = l.tp;
    d.c_out = dW;
    d.ld_c = H;
    d.accumulate = accumulate_dw ? 1 : 0;
    e = launch_gemm_store(d, s);
  }
  return e;
}

cudaError_t launch_transpose_quantize(const uint16_t* in, int64_t rows, int64_t cols, int64_t ld_in,
                                      uint8_t* codes, float* scales, int64_t ld_out, bool pow2,
                                      cudaStream_t s) {
  if (rows == 0 || cols == 0) return cudaSuccess;
  if (cols % 8 != 0 || ld_in % 8 != 0 || ld_out % kQT != 0 || ld_out < rows) return cudaErrorInvalidValue;
  const int64_t gx = ld_out / kQT, gy = (cols + kQT - 1) / kQT;
  if (gx > 0x7FFFFFFF || gy > 65535) return cudaErrorInvalidValue;
  transpose_quantize_kernel<<<dim3(static_cast<unsigned>(gx), static_cast<unsigned>(gy)), 256, 0, s>>>(
      in, rows, cols, ld_in, codes, scales, ld_out, pow2 ? 1 : 0);
  return cudaGetLastError();
}

uint32_t backward_status_take() {
  uint32_t v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, d_status, sizeof(v)) != cudaSuccess) return 0;
  cudaMemcpyToSymbol(d_status, &z, sizeof(z));
  return v;
}

}  // namespace fp8rl
