// Parameters, tile order and epilogues of the lm_head GEMM kernels
// (gemm.cu).
#pragma once

#include <cmath>

#include "common.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

constexpr int CHUNK = 128;        // vocabulary columns per LSE partial
constexpr float kLog2e = 1.4426950408889634f;

enum {
  kTensor = FP8RL_GRAN_TENSOR,
  kRow = FP8RL_GRAN_ROWWISE,
  kBlock = FP8RL_GRAN_BLOCK,
  kUe8m0 = FP8RL_GRAN_BLOCK_UE8M0,  // block layout, power-of-two scales applied by the MMA
  kBf16 = 16
};
static_assert(kBf16 == kGemmBf16, "BF16 mode id shared with the host interface");
// Epilogues: streaming LSE partials + target logit; dense dlogits rows (fp32);
// dlogits of every token E4M3-quantised in both orientations, the A operands
// of the two FP8 backward contractions (gemm.cu); plain store of the fp32
// accumulators (optionally added to what is there).
enum { kEpiLse = 0, kEpiDlogits = 1, kEpiDenseFp8 = 2, kEpiStore = 3 };

struct Params {
  const float* a_scales;
  const float* b_scales;
  const int32_t* targets;
  float2* partials;
  float* zy;
  const float* lse;
  const float* grad;
  float* out;
  uint8_t* pq_out;   // kEpiDenseFp8: P codes [M][ld_pq], 1x128 blocks along N
  float* pq_scales;  //   [ld_pq / 128][M]
  uint8_t* ptq_out;  //   P^T codes [N][ld_ptq], 128 x 128 blocks
  float* ptq_scales; //   [ld_ptq / 128][N] (each block's scale on its 128 rows)
  int64_t ld_pq, ld_ptq;
  float* c_out;      // kEpiStore: fp32 [M][ld_c]
  int64_t ld_c;
  int accumulate;
  int p_pow2;        // kEpiDenseFp8: power-of-two scales for P and P^T
  int M, N, K;
  int num_m, num_n, num_kb;
  int band_m;  // row blocks per band of the tile order
  int n_chunks;
  const uint8_t* sf_a;  // UE8M0 mode: E8M0 scale images [num_m][num_kg][512 B]
  const uint8_t* sf_b;  //   [num_n][num_kg][1024 B]
  int num_kg;           //   groups of four K blocks
  uint64_t wait_limit_ns;
};

// Tile order: bands of band_m row blocks, and within a band the row block
// varies fastest.  For the scoring GEMM (band of 64 token blocks) the 152
// tiles in flight then share one or two vocabulary tiles and a band of h codes
// small enough to stay in L2, so the lm_head codes are read once per band and
// h codes about once.  The backward contractions have only 16 column tiles
// (N = H) and long rows: a band of 16 row blocks keeps about half of them in
// flight per row block, which roughly halves the re-reads of the A operand
// against 64 at the cost of more passes over the B operand.
constexpr int kBandM = 64;
constexpr int kBandStore = 16;
__device__ __forceinline__ void tile_coords(int tile, const Params& p, int& m_blk, int& n_blk) {
  const int band = tile / (p.band_m * p.num_n);
  const int m_base = band * p.band_m;
  const int band_m = min(p.band_m, p.num_m - m_base);
  const int local = tile - band * p.band_m * p.num_n;
  m_blk = m_base + local % band_m;
  n_blk = local / band_m;
}

// 2^x on the special-function unit with a subnormal result flushed to zero
// (PTX ex2.approx.ftz.f32).  The logsumexp terms are exp(z - max) <= 1 summed
// into a total of at least 1 (the maximum's own term), so a flushed term, below
// 2^-126, changes no bit of the sum.
__device__ __forceinline__ float exp2_ftz(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Running epilogue state of one thread: row `row`, vocabulary columns
// [col0, col0 + 128) consumed 32 at a time (values already scaled).
struct EpiState {
  float m, s, zy;
  int j;     // target column relative to col0 (outside [0, 128): not here)
  float l, g;  // dense dlogits epilogue: lse and dLoss/dlogp of the row
};

template <int EPI>
__device__ __forceinline__ void epi_begin(const Params& p, EpiState& e, int row, int col0) {
  e.m = -INFINITY;
  e.s = 0.f;
  e.zy = 0.f;
  e.j = -1;
  e.l = 0.f;
  e.g = 0.f;
  if (EPI != kEpiStore && row < p.M) {
    const int y = p.targets[row];
    if (y >= 0 && y < p.N) e.j = y - col0;
  }
  // loaded when the tile starts, so their latency hides behind its K loop
  if (EPI == kEpiDenseFp8 && row < p.M) {
    e.l = p.lse[row];
    e.g = p.grad[row];
  }
}

// Columns [col0 + base, col0 + base + 32).
template <int EPI>
__device__ __forceinline__ void epi_consume32(const Params& p, EpiState& e, const float* z, int row,
                                              int col0, int base) {
  const int ncol = p.N - (col0 + base);  // valid columns in this piece (may be <= 0 or >= 32)
  if (ncol <= 0 || row >= p.M) return;
  if (EPI == kEpiLse) {
    float cm = -INFINITY;
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (i < ncol) cm = fmaxf(cm, z[i]);
    const float mn = fmaxf(e.m, cm);
    const float mb = mn * kLog2e;
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (i < ncol) acc += exp2_ftz(fmaf(z[i], kLog2e, -mb));
    e.s = e.s * exp2_ftz((e.m - mn) * kLog2e) + acc;
    e.m = mn;
    const int jj = e.j - base;
    if (jj >= 0 && jj < 32) {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (i == jj) e.zy = z[i];
    }
  } else if (EPI == kEpiDlogits) {
    const float l = p.lse[row], g = p.grad[row];
    float* o = p.out + static_cast<size_t>(row) * p.N + col0 + base;
    const int jj = e.j - base;
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (i < ncol) o[i] = g * ((i == jj ? 1.f : 0.f) - expf(z[i] - l));
  } else {  // kEpiStore
    float* cr = p.c_out + static_cast<size_t>(row) * p.ld_c + col0 + base;  // 16-byte aligned
    if (ncol >= 32) {
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        float4 v = make_float4(z[4 * q], z[4 * q + 1], z[4 * q + 2], z[4 * q + 3]);
        if (p.accumulate) {
          const float4 o = reinterpret_cast<const float4*>(cr)[q];
          v.x += o.x;
          v.y += o.y;
          v.z += o.z;
          v.w += o.w;
        }
        reinterpret_cast<float4*>(cr)[q] = v;
      }
    } else {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (i < ncol) cr[i] = p.accumulate ? cr[i] + z[i] : z[i];
    }
  }
}

// All 128 columns of a thread at once (block and UE8M0 scaling, which hold the
// whole row of the tile half in registers): the same (max, sum exp) and z_y as
// four epi_consume32 calls, with one maximum and one rescale instead of four
// and no per-column bounds tests when the whole chunk lies inside [0, N).
template <int EPI>
__device__ __forceinline__ void epi_consume128(const Params& p, EpiState& e, const float* z, int row, int col0) {
  if (EPI != kEpiLse || p.N - col0 < CHUNK || row >= p.M) {
#pragma unroll
    for (int c = 0; c < CHUNK / 32; ++c) epi_consume32<EPI>(p, e, z + c * 32, row, col0, c * 32);
    return;
  }
  float m4[4] = {z[0], z[1], z[2], z[3]};
#pragma unroll
  for (int i = 4; i < CHUNK; i += 4) {
    m4[0] = fmaxf(m4[0], z[i]);
    m4[1] = fmaxf(m4[1], z[i + 1]);
    m4[2] = fmaxf(m4[2], z[i + 2]);
    m4[3] = fmaxf(m4[3], z[i + 3]);
  }
  const float mn = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
  const float mb = mn * kLog2e;
  float a4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int i = 0; i < CHUNK; ++i) a4[i & 3] += exp2_ftz(fmaf(z[i], kLog2e, -mb));
  e.s = (a4[0] + a4[1]) + (a4[2] + a4[3]);
  e.m = mn;
  if (e.j >= 0 && e.j < CHUNK) {
#pragma unroll
    for (int i = 0; i < CHUNK; ++i)
      if (i == e.j) e.zy = z[i];
  }
}

template <int EPI>
__device__ __forceinline__ void epi_finish(const Params& p, const EpiState& e, int row, int chunk) {
  if (EPI != kEpiLse || row >= p.M || chunk >= p.n_chunks) return;
  p.partials[static_cast<size_t>(chunk) * p.M + row] = make_float2(e.m, e.s);
  if (e.j >= 0 && e.j < CHUNK) p.zy[row] = e.zy;
}


}  // namespace
}  // namespace fp8rl
