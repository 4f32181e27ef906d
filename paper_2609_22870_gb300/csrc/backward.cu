// Backward through the FP8 lm_head: given g_t = dLoss/dlogp_t (the clipped
// surrogate's gradient) and the forward pass's lse, the chain rule through the
// log-softmax gives dLoss/dz[t][v] = g_t (1{v == y_t} - exp(z[t][v] - lse_t)),
// and through z = h W^T the two contractions
//   dh = P W  ([T][V] x [V][H]),     dW = P^T h  ([V][T] x [T][H]).
// The quantisers pass the gradient straight through, so the contractions take
// the bf16 operands.  Steps, all on the caller's stream:
//   1. the FP8 GEMM recomputes z tile by tile and its epilogue writes P in
//      bf16 twice, [T][V] and [V][T] (logits themselves are never stored);
//   2. W and h are transposed to [H][V] and [H][T] (K-major B operands);
//   3. the tcgen05 BF16 GEMM forms dh (K = V) and dW (K = T) into fp32.
#include "common.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

constexpr int kTile = 32;

// out[c][r] = in[r][c] for a bf16 matrix [rows][cols]: 32 x 32 tiles through
// shared memory (padded against bank conflicts), 32 x 8 threads, four
// elements a thread each way.
__global__ void __launch_bounds__(256) transpose_bf16_kernel(const uint16_t* __restrict__ in,
                                                             int64_t rows, int64_t cols, int64_t ld_in,
                                                             uint16_t* __restrict__ out, int64_t ld_out) {
  __shared__ uint16_t tile[kTile][kTile + 2];
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kTile;
  const int64_t r0 = static_cast<int64_t>(blockIdx.y) * kTile;
  const int tx = threadIdx.x, ty = threadIdx.y;
#pragma unroll
  for (int k = 0; k < kTile; k += 8) {
    const int64_t r = r0 + ty + k, c = c0 + tx;
    if (r < rows && c < cols) tile[ty + k][tx] = in[r * ld_in + c];
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < kTile; k += 8) {
    const int64_t c = c0 + ty + k, r = r0 + tx;
    if (c < cols && r < rows) out[c * ld_out + r] = tile[tx][ty + k];
  }
}

}  // namespace

BwdLayout bwd_layout(int64_t T, int64_t H, int64_t V) {
  BwdLayout l;
  l.vp = (V + 7) / 8 * 8;  // bf16 row strides must be multiples of 16 bytes (TMA)
  l.tp = (T + 7) / 8 * 8;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes, 256);
    return at;
  };
  l.p = take(static_cast<size_t>(T) * l.vp * 2);
  l.pt = take(static_cast<size_t>(V) * l.tp * 2);
  l.wt = take(static_cast<size_t>(H) * l.vp * 2);
  l.ht = take(static_cast<size_t>(H) * l.tp * 2);
  l.total = off;
  return l;
}

cudaError_t launch_lm_head_backward(const uint8_t* hc, const float* hs, const uint8_t* wc,
                                    const float* wsc, int gran, int64_t T, int64_t H, int64_t V,
                                    const int32_t* targets, const float* lse, const float* grad,
                                    const uint16_t* h, const uint16_t* W, float* dh, float* dW,
                                    int accumulate_dw, void* ws, cudaStream_t s) {
  const BwdLayout l = bwd_layout(T, H, V);
  char* base = static_cast<char*>(ws);
  uint16_t* P = reinterpret_cast<uint16_t*>(base + l.p);
  uint16_t* Pt = reinterpret_cast<uint16_t*>(base + l.pt);
  uint16_t* Wt = reinterpret_cast<uint16_t*>(base + l.wt);
  uint16_t* Ht = reinterpret_cast<uint16_t*>(base + l.ht);
  // 1. recompute z (FP8), write P = dLoss/dz in bf16, both orientations
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
  a.p_out = P;
  a.pt_out = Pt;
  a.ld_p = l.vp;
  a.ld_pt = l.tp;
  cudaError_t e = launch_gemm_dense_dlogits(a, s);
  if (e != cudaSuccess) return e;
  if (dh) {  // 2./3. dh[T][H] = P[T][V] . W[V][H]: B operand W^T [H][V]
    e = launch_transpose_bf16(W, V, H, H, Wt, l.vp, s);
    if (e != cudaSuccess) return e;
    GemmArgs d{};
    d.a_codes = P;
    d.b_codes = Wt;
    d.gran = kGemmBf16;
    d.M = T;
    d.N = H;
    d.K = V;
    d.lda = l.vp;
    d.ldb = l.vp;
    d.c_out = dh;
    d.ld_c = H;
    e = launch_gemm_store(d, s);
    if (e != cudaSuccess) return e;
  }
  if (dW) {  // dW[V][H] = P^T[V][T] . h[T][H]: B operand h^T [H][T]
    e = launch_transpose_bf16(h, T, H, H, Ht, l.tp, s);
    if (e != cudaSuccess) return e;
    GemmArgs d{};
    d.a_codes = Pt;
    d.b_codes = Ht;
    d.gran = kGemmBf16;
    d.M = V;
    d.N = H;
    d.K = T;
    d.lda = l.tp;
    d.ldb = l.tp;
    d.c_out = dW;
    d.ld_c = H;
    d.accumulate = accumulate_dw;
    e = launch_gemm_store(d, s);
  }
  return e;
}

cudaError_t launch_transpose_bf16(const uint16_t* in, int64_t rows, int64_t cols, int64_t ld_in,
                                  uint16_t* out, int64_t ld_out, cudaStream_t s) {
  if (rows == 0 || cols == 0) return cudaSuccess;
  const int64_t gx = (cols + kTile - 1) / kTile, gy = (rows + kTile - 1) / kTile;
  if (gx > 0x7FFFFFFF || gy > 65535) return cudaErrorInvalidValue;
  transpose_bf16_kernel<<<dim3(static_cast<unsigned>(gx), static_cast<unsigned>(gy)), dim3(kTile, 8), 0, s>>>(
      in, rows, cols, ld_in, out, ld_out);
  return cudaGetLastError();
}

}  // namespace fp8rl
