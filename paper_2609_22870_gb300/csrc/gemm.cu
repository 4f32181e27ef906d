// a3: FP8 lm_head GEMM on the tcgen05 tensor cores with a streaming
// logsumexp + target-gather epilogue (§2.1 ratio, Eq. 3 scaling); the merge of
// the per-chunk partials into log-probs and ratios (a4) is in combine.cu.
//
// z[t][v] = sum_k S_h S_W q_h[t][k] q_W[v][k] is never stored.  Each CTA owns
// persistent 128 (tokens) x 256 (vocab) output tiles:
//   warp 0      TMA producer: 128x128 A tile + 256x128 B tile per stage, 128B
//               swizzle, 4-stage shared-memory ring guarded by mbarriers;
//   warp 1      MMA issuer: tcgen05.mma kind::f8f6f4 M=128 N=256 K=32, fp32
//               accumulator in TMEM (two 256-column buffers);
//   warp 2      block scaling only: stages the activation and weight scales
//               of four K blocks per slot into a shared-memory ring, so the
//               epilogue never waits on global loads and meets one barrier per
//               four K blocks;
//   warp 3      idle (it completes the first warpgroup, whose register budget
//               is lowered to 56 so the epilogue can hold 224);
//   warps 4..11 epilogue: tcgen05.ld of the accumulator, one thread per token
//               row and 128-column half, scales applied, then the running
//               (max, sum exp) of its 128 columns and z[t][y_t] if y_t falls in
//               them.  One (max, sum) pair per token and 128-wide vocabulary
//               chunk goes to the workspace; nothing of size T x V does.
// Per-tensor and per-row scales factor out of the K sum, so the accumulator
// runs over the whole K in TMEM and is scaled once.  The BF16 shadow pass of §4
// (reference log-probs from the unquantised operands) runs the same kernel with
// tcgen05.mma kind::f16 on bf16 tiles (64 elements = 128 bytes per row and
// stage, so the shared-memory layout is the FP8 one) and no scales.  Block scales (1x128 for h,
// 128x128 for W) change every 128-wide K block: the MMA writes each K block's
// partial product into one of the two TMEM buffers and the epilogue promotes
// it, acc += S_h[t][kb] S_W[vb][kb] * partial, into registers while the MMA
// fills the other buffer.
// Power-of-two block scales (the UE8M0 variant) go to the tensor cores instead:
// tcgen05.mma kind::mxf8f6f4 multiplies each 32-wide K step by E8M0 scale
// factors it reads from TMEM, so one accumulator runs over the whole K and the
// epilogue only reads it once per tile.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cmath>

#include "common.cuh"
#include "e4m3_encode.cuh"
#include "gemm_epi.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

__device__ uint32_t d_status;

constexpr int BM = 128;           // tokens per tile (TMEM lanes)
constexpr int BN = 256;           // vocabulary columns per tile (MMA N)
constexpr int BK = 128;           // K bytes per stage (one 128B swizzle row)
constexpr int STAGES = 4;
constexpr int EPI_WARPS = 8;
constexpr int EPI_WARP0 = 4;      // first epilogue warp (start of warpgroup 1)
constexpr int THREADS = 128 + EPI_WARPS * 32;
constexpr int CTRL_REGS = 56;     // register budget of warpgroup 0 (producer, MMA)
constexpr int EPI_REGS = 224;     // register budget of the two epilogue warpgroups
constexpr uint32_t A_BYTES = BM * BK;
constexpr uint32_t B_BYTES = BN * BK;
constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
constexpr uint32_t TMEM_COLS = 2 * BN;
constexpr int SC_SLOTS = 4;                       // scale ring depth (slots)
constexpr int SC_KB = 4;                          // K blocks per slot
constexpr uint32_t SC_KB_FLOATS = BM + 4;         // 128 activation + 2 weight (+2 pad)
constexpr uint32_t SC_SLOT_FLOATS = SC_KB * SC_KB_FLOATS;
constexpr uint32_t SC_BYTES = SC_SLOTS * SC_SLOT_FLOATS * 4;
// UE8M0 (hardware block scaling) mode: the E8M0 scale factors come as images
// in global memory (ue8m0_pack_kernel), one per group of four K blocks and
// 128-row token block or 256-row vocabulary tile, and the producer loads a
// group's images with the stage of its first K block.  An image is 32 lanes x
// 16 bytes: row i of the block in lane i % 32, word i / 32, and byte q of the
// word the scale of K block 4g + q.  One image covers the 128 token rows, two
// the 256 vocabulary rows.
constexpr int SF_KB = 4;                          // K blocks per image group
constexpr uint32_t SF_IMG_BYTES = 512;
constexpr uint32_t SF_GROUP_BYTES = 3 * SF_IMG_BYTES;
constexpr uint32_t SF_BYTES = STAGES * SF_GROUP_BYTES;
// In TMEM the mode keeps one 256-column accumulator (columns 0..255) and a
// ring of scale factors from column 256: per group 4 columns for the rows of A
// and 8 for those of B (entry i in lane i % 32 of every lane quarter, column
// i / 32), 16 groups deep.
constexpr uint32_t SF_TCOL0 = 256;
constexpr uint32_t SF_TCOLS = 12;
constexpr int SF_TRING = 16;
template <int MODE>
constexpr uint32_t ring_bytes() { return MODE == kUe8m0 ? SF_BYTES : SC_BYTES; }
template <int MODE>
constexpr size_t smem_bytes() { return 1024 + STAGES * STAGE_BYTES + ring_bytes<MODE>() + 512; }
constexpr uint64_t kDrainNs = 1000000000ull;
// Exchange slots of the dense FP8 epilogue's 128 x 128 block maxima: an
// epilogue warp runs at most two tiles ahead of another (tile i + 2 needs the
// accumulator buffer that every warp released at tile i), so four slots are
// never reused while a slower warp still reads one.
constexpr int XSLOTS = 4;

__device__ __forceinline__ void flag(uint32_t bits) { atomicOr(&d_status, bits); }

// E8M0 byte of a power-of-two float32 scale (its biased exponent; 2^-127,
// a subnormal float32, is byte 0).  A scale that is not a positive power of
// two in E8M0's range is bad input: NaN byte 0xFF, status flagged.
__device__ __forceinline__ uint32_t e8m0_byte(float s) {
  const uint32_t b = __float_as_uint(s);
  if (b == 0x00400000u) return 0;
  const uint32_t e = b >> 23;
  if ((b & 0x807FFFFFu) != 0 || e == 0 || e >= 255) {
    flag(kErrDevice);
    return 0xFFu;
  }
  return e;
}

// Bulk copy global -> shared of `bytes` (a multiple of 16, both addresses
// 16-byte aligned), completing as transaction bytes on mbarrier `bar`.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// Shared-memory descriptor of a 32-row x 16-byte image without swizzle
// (8-row x 16-byte core matrices, 128 bytes apart), the source of a
// 32x128b tcgen05.cp.
__device__ __forceinline__ uint64_t smem_desc_plain(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(128u >> 4) << 16;
  d |= static_cast<uint64_t>(128u >> 4) << 32;
  d |= static_cast<uint64_t>(1u) << 46;
  return d;
}

// Copies a 32-row x 128-bit image from shared memory to TMEM columns
// [taddr, taddr + 4) of lanes 0..31, repeated in every lane quarter; issued by
// one elected lane of a converged warp, in order with its MMAs.
__device__ __forceinline__ void tmem_cp_32x128b_x4_elect(uint32_t taddr, uint64_t sdesc) {
  asm volatile(
      "{\n\t.reg .pred e;\n\t"
      "elect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;\n\t}" ::"r"(taddr),
      "l"(sdesc)
      : "memory");
}

// D (+)= (A x SFA) * (B x SFB)^T with E8M0 scale factors per 32-wide K step
// (kind::mxf8f6f4, E4M3 operands): sfa / sfb are TMEM addresses of the scale
// vectors, idesc selects the byte of each word; warp-converged.
__device__ __forceinline__ void mma_mx_e4m3_elect(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                                  uint32_t idesc, uint32_t sfa, uint32_t sfb,
                                                  uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p, e;\n\t"
      "setp.ne.b32 p, %6, 0;\n\t"
      "elect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], %1, %2, %3, [%4], [%5], p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(sfa), "r"(sfb), "r"(accumulate)
      : "memory");
}

// Instruction descriptor of the block-scaled MMA: E4M3 A and B, K-major,
// E8M0 scale factors (bit 23), N >> 3 at bit 17, M >> 7 at bit 27; the scale
// byte of B at bits 4-5 and of A at bits 29-30.
__host__ __device__ constexpr uint32_t idesc_mx_e4m3(uint32_t M, uint32_t N) {
  return ((N >> 3) << 17) | (1u << 23) | ((M >> 7) << 27);
}

// E4M3 codes Q_FP8(fl32(v_i / S)) of 128 floats, four per word (byte i % 4 of
// word i / 4), in the packed arithmetic of the quantiser.  With pow2 (S a
// power of two in [2^-127, 2^120]) 1 / S is exact and so is v * (1 / S)
// wherever it is at least 2^-126; below that both forms give code 0 of v's
// sign, so one packed multiply replaces the corrected quotient.
__device__ __forceinline__ void encode128(const float* v, float s, uint32_t (&w)[32], bool pow2) {
  if (pow2) {
    const float r = __frcp_rn(s);
    const uint64_t r2 = f32x2(r, r);
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      uint64_t q0, q1;
      asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(q0) : "l"(f32x2(v[4 * i], v[4 * i + 1])), "l"(r2));
      asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(q1) : "l"(f32x2(v[4 * i + 2], v[4 * i + 3])), "l"(r2));
      w[i] = cvt_e4m3x2(q0) | (cvt_e4m3x2(q1) << 16);
    }
    return;
  }
  const E4M3Enc e = e4m3_encoder(s);
  if (!e.divide) {
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const uint32_t a = cvt_e4m3x2(neg_quotient2(f32x2(v[4 * i], v[4 * i + 1]), e));
      const uint32_t b = cvt_e4m3x2(neg_quotient2(f32x2(v[4 * i + 2], v[4 * i + 3]), e));
      w[i] = (a | (b << 16)) ^ 0x80808080u;  // the quotients were negated
    }
  } else {
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const uint32_t a = static_cast<uint32_t>(__nv_cvt_float2_to_fp8x2(
          make_float2(__fdiv_rn(v[4 * i], s), __fdiv_rn(v[4 * i + 1], s)), __NV_SATFINITE, __NV_E4M3));
      const uint32_t b = static_cast<uint32_t>(__nv_cvt_float2_to_fp8x2(
          make_float2(__fdiv_rn(v[4 * i + 2], s), __fdiv_rn(v[4 * i + 3], s)), __NV_SATFINITE, __NV_E4M3));
      w[i] = a | (b << 16);
    }
  }
}

// S = fl32(amax / 448), 1 for an all-zero block (NaN amax gives NaN).
__device__ __forceinline__ float scale_of(float amax) { return amax == 0.f ? 1.f : __fdiv_rn(amax, kE4M3Max); }

// max that propagates NaN (a NaN block maximum marks the block's scale NaN).
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

// Dense dLoss/dz of one thread's 128 columns (row `row`, columns col0 ..
// col0 + 127; z the scaled logits), quantised for the FP8 backward:
//   P[t][v] = g_t (1{v == y_t} - exp(z[t][v] - lse_t))   (float32, the
//   exponential as exp2(z log2(e) - lse log2(e)) with one fused multiply-add)
//   codes of P with this row's 1x128 block scale        -> pq_out / pq_scales
//   codes of P with the 128 x 128 block scale of the tile half (the max over
//   the four warps holding its 128 rows, exchanged through shared memory
//   with a bounded wait), stored transposed         -> ptq_out / ptq_scales
// With p.p_pow2 both scales are rounded up to powers of two and floored at
// 2^-127, the scale format of the block-scaled MMA that then runs the
// contractions.  Rows past M and columns past N hold 0 (the K padding of
// the contractions).  Returns false if the exchange wait expired.
__device__ __forceinline__ float p_scale(float amax, bool pow2) {
  const float s = scale_of(amax);
  return pow2 ? e8m0_floor(pow2_ceil(s)) : s;
}

__device__ __forceinline__ bool dense_fp8_epilogue(const Params& p, const EpiState& es, float* z, int row,
                                                   int col0, int m_blk, int rit, int half, int quarter,
                                                   int lane, int tcount, uint64_t* blk_bar, uint32_t* blk_max,
                                                   uint64_t lim, const volatile int* abort_flag) {
  const bool pow2 = p.p_pow2 != 0;
  const int ncol = min(CHUNK, p.N - col0);
  const bool row_ok = row < p.M;
  const float g = es.g;
  const float lb = es.l * kLog2e;
  float amax = 0.f;
  const bool here = es.j >= 0 && es.j < CHUNK;
  if (__all_sync(0xffffffffu, row_ok && !here) && ncol == CHUNK) {
    // the common case: every row of the warp valid, no target column here
    const float ng = -g;
#pragma unroll
    for (int i = 0; i < CHUNK; ++i) {
      const float v = ng * exp2f(fmaf(z[i], kLog2e, -lb));
      z[i] = v;
      amax = fmax_nan(amax, fabsf(v));
    }
  } else {
#pragma unroll
    for (int i = 0; i < CHUNK; ++i) {
      const float v = (row_ok && i < ncol) ? g * ((i == es.j ? 1.f : 0.f) - exp2f(fmaf(z[i], kLog2e, -lb))) : 0.f;
      z[i] = v;
      amax = fmax_nan(amax, fabsf(v));
    }
  }
  uint32_t w[32];
  if (row_ok && col0 < p.ld_pq) {  // the row's block along N (K of the dh contraction)
    const float s = p_scale(amax, pow2);
    encode128(z, s, w, pow2);
    uint4* dst = reinterpret_cast<uint4*>(p.pq_out + static_cast<size_t>(row) * p.ld_pq + col0);
#pragma unroll
    for (int q = 0; q < 8; ++q) dst[q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
    p.pq_scales[static_cast<size_t>(col0 / CHUNK) * p.M + row] = s;
  }
  // 128 x 128 block maximum: non-negative floats (and NaN above them) order
  // like their bit patterns
  const uint32_t wmax = __reduce_max_sync(0xffffffffu, __float_as_uint(amax));
  const int slot = tcount % XSLOTS;
  const uint32_t par = static_cast<uint32_t>(tcount / XSLOTS) & 1u;
  uint32_t* bm = blk_max + (slot * 2 + half) * 4;
  const uint32_t bar = smem_u32(&blk_bar[slot * 2 + half]);
  if (lane == 0) {
    bm[quarter] = wmax;
    mbar_arrive(bar);
  }
  if (!__all_sync(0xffffffffu, mbar_wait(bar, par, lim, abort_flag))) return false;
  const uint32_t bmax = max(max(bm[0], bm[1]), max(bm[2], bm[3]));
  if (ncol <= 0) return true;
  const float sb = p_scale(__uint_as_float(bmax), pow2);
  encode128(z, sb, w, pow2);
  // lanes are consecutive tokens; a 4 x 4 byte transpose within each group of
  // four lanes (two exchanges) leaves lane 4a + j with column 4k + j of rows
  // 4a .. 4a + 3, so each store writes four bytes and each column of P^T gets
  // 32 contiguous bytes per warp
  const int j = lane & 3;
  const size_t ld = static_cast<size_t>(p.ld_ptq);
  uint8_t* dst = p.ptq_out + static_cast<size_t>(col0 + j) * ld + (row - j);
#pragma unroll
  for (int k = 0; k < CHUNK / 4; ++k) {
    // round 1 (lanes j, j ^ 1): even lanes keep bytes 0, 2 and take the
    // partner's; odd lanes keep 1, 3
    const uint32_t o1 = __shfl_xor_sync(0xffffffffu, w[k], 1);
    const uint32_t r1 = (j & 1) ? __byte_perm(o1, w[k], 0x7351) : __byte_perm(w[k], o1, 0x6240);
    // round 2 (lanes j, j ^ 2): lanes 0, 1 keep their low halves
    const uint32_t o2 = __shfl_xor_sync(0xffffffffu, r1, 2);
    const uint32_t t = (j & 2) ? __byte_perm(o2, r1, 0x7632) : __byte_perm(r1, o2, 0x5410);
    if (4 * k + j < ncol) *reinterpret_cast<uint32_t*>(dst + static_cast<size_t>(4 * k) * ld) = t;
  }
  if (rit < ncol) p.ptq_scales[static_cast<size_t>(m_blk) * p.N + col0 + rit] = sb;
  return true;
}

template <int MODE, int EPI>
__global__ void __launch_bounds__(THREADS, 1)
    fp8_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* smA = smem;
  uint8_t* smB = smem + STAGES * A_BYTES;
  float* sc_ring = reinterpret_cast<float*>(smB + STAGES * B_BYTES);  // [SC_SLOTS][132]
  uint8_t* sf_img = smB + STAGES * B_BYTES;  // UE8M0 mode: [STAGES][3 images]
  uint64_t* bars = reinterpret_cast<uint64_t*>(smB + STAGES * B_BYTES + ring_bytes<MODE>());
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* acc_full = bars + 2 * STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* sc_full = acc_empty + 2;
  uint64_t* sc_empty = sc_full + SC_SLOTS;
  uint64_t* done = sc_empty + SC_SLOTS;
  uint64_t* blk_bar = done + 1;  // dense FP8 epilogue: [XSLOTS][2 halves]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(blk_bar + XSLOTS * 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  uint32_t* blk_max = tmem_holder + 2;  // [XSLOTS][2 halves][4 warps] float bits

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&acc_full[b]), 1);
      mbar_init(smem_u32(&acc_empty[b]), EPI_WARPS);
    }
    for (int i = 0; i < SC_SLOTS; ++i) {
      mbar_init(smem_u32(&sc_full[i]), 32);
      mbar_init(smem_u32(&sc_empty[i]), EPI_WARPS);
    }
    mbar_init(smem_u32(done), 1);
    for (int i = 0; i < XSLOTS * 2; ++i) mbar_init(smem_u32(&blk_bar[i]), 4);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_holder), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const int total = p.num_m * p.num_n;
  const uint64_t lim = p.wait_limit_ns;

  if (warp < EPI_WARP0) {
   warpgroup_reg_dealloc<CTRL_REGS>();
   if (warp == 0) {
    // ------------------------------------------------------------ producer
    // the whole warp runs the loop (uniform control flow); one elected lane
    // issues the barrier arrive and the two TMA loads of each stage
    int stage = 0;
    uint32_t phase = 0;
    uint32_t armed = 0, armed_phase = 0;  // bit s: stage s loaded / its parity
    bool ok = true;
    for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
      int m_blk, n_blk;
      tile_coords(tile, p, m_blk, n_blk);
      const int m0 = m_blk * BM, n0 = n_blk * BN;
      for (int kb = 0; kb < p.num_kb; ++kb) {
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&empty[stage]), phase ^ 1, lim, abort_flag));
        if (!ok) break;
        if (elect_one()) {
          // UE8M0 mode: the first K block of each group also brings the
          // group's scale-factor images
          const bool sf = MODE == kUe8m0 && kb % SF_KB == 0;
          mbar_arrive_expect_tx(smem_u32(&full[stage]), STAGE_BYTES + (sf ? SF_GROUP_BYTES : 0u));
          // K coordinate in elements: 128 E4M3 or 64 BF16 per 128-byte row
          const int kx = kb * ((MODE == kBf16) ? BK / 2 : BK);
          tma_load_2d(smem_u32(smA + stage * A_BYTES), &tmA, smem_u32(&full[stage]), kx, m0);
          tma_load_2d(smem_u32(smB + stage * B_BYTES), &tmB, smem_u32(&full[stage]), kx, n0);
          if (sf) {
            const size_t g = static_cast<size_t>(kb / SF_KB);
            const uint32_t dst = smem_u32(sf_img + stage * SF_GROUP_BYTES);
            bulk_load(dst, p.sf_a + (static_cast<size_t>(m_blk) * p.num_kg + g) * SF_IMG_BYTES, SF_IMG_BYTES,
                      smem_u32(&full[stage]));
            bulk_load(dst + SF_IMG_BYTES, p.sf_b + (static_cast<size_t>(n_blk) * p.num_kg + g) * 2 * SF_IMG_BYTES,
                      2 * SF_IMG_BYTES, smem_u32(&full[stage]));
          }
        }
        __syncwarp();
        armed |= 1u << stage;
        armed_phase = (armed_phase & ~(1u << stage)) | (phase << stage);
        if (++stage == STAGES) {
          stage = 0;
          phase ^= 1;
        }
      }
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      flag(kErrTimeout);
    }
    // no copy may still be in flight when the CTA exits
    for (int s = 0; s < STAGES; ++s)
      if (armed & (1u << s)) mbar_wait(smem_u32(&full[s]), (armed_phase >> s) & 1, kDrainNs, nullptr);
   } else if (warp == 2 && MODE == kBlock) {
    // ------------------------------------------------------------ scale loader
    // per K block: the 128 activation scales S_h[kb][m0 .. m0+127] and the
    // scales of the two weight blocks the tile spans, into ring slot `slot`
    int slot = 0;
    uint32_t sphase = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
      int m_blk, n_blk;
      tile_coords(tile, p, m_blk, n_blk);
      const int m0 = m_blk * BM;
      const int wb0 = 2 * n_blk;
      for (int kg = 0; kg < p.num_kb; kg += SC_KB) {
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&sc_empty[slot]), sphase ^ 1, lim, abort_flag));
        if (!ok) break;
        const int nkb = min(SC_KB, p.num_kb - kg);
        for (int q = 0; q < nkb; ++q) {
          const int kb = kg + q;
          const uint32_t dst = smem_u32(sc_ring + slot * SC_SLOT_FLOATS + q * SC_KB_FLOATS);
          const float* src = p.a_scales + static_cast<size_t>(kb) * p.M;
          // asynchronous 4-byte copies: the warp never waits for the data, the
          // barrier completes when every lane's copies have landed
#pragma unroll
          for (int j = 0; j < BM / 32; ++j) {
            const int r = m0 + j * 32 + lane;
            if (r < p.M) cp_async_4(dst + (j * 32 + lane) * 4, src + r);
          }
          if (lane < 2 && wb0 + lane < p.n_chunks)
            cp_async_4(dst + (BM + lane) * 4, p.b_scales + static_cast<size_t>(wb0 + lane) * p.num_kb + kb);
        }
        cp_async_mbar_arrive(smem_u32(&sc_full[slot]));
        if (++slot == SC_SLOTS) {
          slot = 0;
          sphase ^= 1;
        }
      }
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      flag(kErrTimeout);
    }
    asm volatile("cp.async.wait_all;" ::: "memory");  // no copy in flight at exit
   } else if (warp == 1 && MODE == kUe8m0) {
    // ------------------------------------------------------------ MMA issuer (UE8M0)
    // one accumulator over all of K; at the first K block of each group the
    // group's scale images are copied from the stage into the TMEM ring (in
    // order with the MMAs that read them, so the stage's release covers the
    // copy too), and each K block's four block-scaled MMAs select byte
    // kb % 4 of the scale words
    int stage = 0, gcount = 0;
    uint32_t phase = 0, aphase = 0;
    uint32_t sf = tmem_base + SF_TCOL0;
    constexpr uint32_t idesc = idesc_mx_e4m3(BM, BN);
    bool ok = true;
    for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
      ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&acc_empty[0]), aphase ^ 1, lim, abort_flag));
      if (!ok) break;
      tc_fence_after();
      for (int kb = 0; kb < p.num_kb; ++kb) {
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&full[stage]), phase, lim, abort_flag));
        if (!ok) break;
        tc_fence_after();
        const uint32_t q = static_cast<uint32_t>(kb % SF_KB);
        if (q == 0) {
          sf = tmem_base + SF_TCOL0 + static_cast<uint32_t>(gcount % SF_TRING) * SF_TCOLS;
          ++gcount;
          const uint32_t img = smem_u32(sf_img + stage * SF_GROUP_BYTES);
          tmem_cp_32x128b_x4_elect(sf, smem_desc_plain(img));
          tmem_cp_32x128b_x4_elect(sf + 4, smem_desc_plain(img + SF_IMG_BYTES));
          tmem_cp_32x128b_x4_elect(sf + 8, smem_desc_plain(img + 2 * SF_IMG_BYTES));
        }
        const uint64_t adesc = smem_desc_sw128(smem_u32(smA + stage * A_BYTES));
        const uint64_t bdesc = smem_desc_sw128(smem_u32(smB + stage * B_BYTES));
        const uint32_t id = idesc | (q << 29) | (q << 4);
#pragma unroll
        for (int k = 0; k < BK / 32; ++k)
          mma_mx_e4m3_elect(tmem_base, adesc + 2 * k, bdesc + 2 * k, id, sf, sf + 4, kb > 0 || k > 0);
        mma_commit_elect(smem_u32(&empty[stage]));
        if (++stage == STAGES) {
          stage = 0;
          phase ^= 1;
        }
      }
      if (!ok) break;
      mma_commit_elect(smem_u32(&acc_full[0]));
      aphase ^= 1;
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      flag(kErrTimeout);
    }
    mma_commit_elect(smem_u32(done));
    mbar_wait(smem_u32(done), 0, kDrainNs, nullptr);
   } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    // whole warp converged; elect.sync picks the lane that issues each
    // tcgen05.mma / tcgen05.commit
    int stage = 0, ab = 0;
    uint32_t phase = 0, aphase = 0;
    constexpr uint32_t idesc = (MODE == kBf16) ? idesc_bf16_f32(BM, BN) : idesc_e4m3_f32(BM, BN);
    bool ok = true;
    for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
      if (MODE != kBlock) {
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&acc_empty[ab]), aphase ^ 1, lim, abort_flag));
        if (!ok) break;
        tc_fence_after();
      }
      for (int kb = 0; kb < p.num_kb; ++kb) {
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&full[stage]), phase, lim, abort_flag));
        if (!ok) break;
        if (MODE == kBlock) {
          ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&acc_empty[ab]), aphase ^ 1, lim, abort_flag));
          if (!ok) break;
        }
        tc_fence_after();
        const uint32_t d = tmem_base + static_cast<uint32_t>(ab * BN);
        const uint64_t adesc = smem_desc_sw128(smem_u32(smA + stage * A_BYTES));
        const uint64_t bdesc = smem_desc_sw128(smem_u32(smB + stage * B_BYTES));
#pragma unroll
        for (int k = 0; k < BK / 32; ++k) {
          const uint32_t acc = (MODE == kBlock) ? (k > 0) : (kb > 0 || k > 0);
          // +32 bytes along K inside the swizzled 128-byte row (32 FP8 or 16 BF16 elements)
          if (MODE == kBf16) mma_bf16_elect(d, adesc + 2 * k, bdesc + 2 * k, idesc, acc);
          else mma_f8f6f4_elect(d, adesc + 2 * k, bdesc + 2 * k, idesc, acc);
        }
        mma_commit_elect(smem_u32(&empty[stage]));
        if (MODE == kBlock) {
          mma_commit_elect(smem_u32(&acc_full[ab]));
          ab ^= 1;
          if (ab == 0) aphase ^= 1;
        }
        if (++stage == STAGES) {
          stage = 0;
          phase ^= 1;
        }
      }
      if (!ok) break;
      if (MODE != kBlock) {
        mma_commit_elect(smem_u32(&acc_full[ab]));
        ab ^= 1;
        if (ab == 0) aphase ^= 1;
      }
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      flag(kErrTimeout);
    }
    // every MMA issued above has completed once this commit lands
    mma_commit_elect(smem_u32(done));
    mbar_wait(smem_u32(done), 0, kDrainNs, nullptr);
   }
  } else {
    warpgroup_reg_alloc<EPI_REGS>();
    // ------------------------------------------------------------ epilogue
    const int ew = warp - EPI_WARP0;
    const int quarter = warp & 3;  // TMEM lanes this warp may access
    const int half = ew >> 2;      // which 128 columns of the 256-wide tile
    const int rit = quarter * 32 + lane;
    const uint32_t t_row = static_cast<uint32_t>(quarter * 32) << 16;
    int ab = 0, sslot = 0, tcount = 0;
    uint32_t aphase = 0, sphase = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x, ++tcount) {
      int m_blk, n_blk;
      tile_coords(tile, p, m_blk, n_blk);
      const int row = m_blk * BM + rit;
      const bool row_ok = row < p.M;
      const int col0 = n_blk * BN + half * CHUNK;
      const int chunk = n_blk * 2 + half;
      EpiState es;
      epi_begin<EPI>(p, es, row, col0);
      if (MODE == kBlock) {
        float2 z2[CHUNK / 2];
#pragma unroll
        for (int i = 0; i < CHUNK / 2; ++i) z2[i] = make_float2(0.f, 0.f);
        for (int kb = 0; kb < p.num_kb; ++kb) {
          // this K block's scales from the ring (staged by the loader warp,
          // SC_KB K blocks per slot: one barrier wait per slot)
          const int q = kb % SC_KB;
          if (q == 0) {
            ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&sc_full[sslot]), sphase, lim, abort_flag));
            if (!ok) break;
          }
          const float* scs = sc_ring + sslot * SC_SLOT_FLOATS + q * SC_KB_FLOATS;
          const float sc = scs[rit] * scs[BM + half];
          if (q == SC_KB - 1 || kb == p.num_kb - 1) {
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&sc_empty[sslot]));
            if (++sslot == SC_SLOTS) {
              sslot = 0;
              sphase ^= 1;
            }
          }
          // the epilogue trails the MMA, so this phase has usually completed
          ok = __all_sync(0xffffffffu, mbar_wait_likely_done(smem_u32(&acc_full[ab]), aphase, lim, abort_flag));
          if (!ok) break;
          tc_fence_after();
          const uint32_t taddr = tmem_base + t_row + static_cast<uint32_t>(ab * BN + half * CHUNK);
          // four 32-column chunks, double-buffered: the load of chunk c + 1
          // is in flight while chunk c is promoted; the TMEM buffer goes back
          // to the MMA as soon as the last chunk has landed in registers
          uint32_t ra[32], rb[32];
          tmem_ld_32x32b_x32_issue(taddr, ra);
          tmem_wait_ld(ra);
#pragma unroll
          for (int c = 0; c < CHUNK / 32; ++c) {
            uint32_t(&cur)[32] = (c & 1) ? rb : ra;
            uint32_t(&nxt)[32] = (c & 1) ? ra : rb;
            if (c + 1 < CHUNK / 32) tmem_ld_32x32b_x32_issue(taddr + (c + 1) * 32, nxt);
            if (c + 1 == CHUNK / 32) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(smem_u32(&acc_empty[ab]));
            }
#pragma unroll
            for (int i = 0; i < 16; ++i)
            {
              // scalar FMAs: the packed f32x2 form measured no faster here
              z2[c * 16 + i].x = fmaf(__uint_as_float(cur[2 * i]), sc, z2[c * 16 + i].x);
              z2[c * 16 + i].y = fmaf(__uint_as_float(cur[2 * i + 1]), sc, z2[c * 16 + i].y);
            }
            if (c + 1 < CHUNK / 32) tmem_wait_ld(nxt);
          }
          ab ^= 1;
          if (ab == 0) aphase ^= 1;
        }
        if (!ok) break;
        float* z = reinterpret_cast<float*>(z2);
        if (EPI == kEpiDenseFp8) {
          ok = dense_fp8_epilogue(p, es, z, row, col0, m_blk, rit, half, quarter, lane, tcount, blk_bar, blk_max,
                                  lim, abort_flag);
          if (!ok) break;
        } else {
          epi_consume128<EPI>(p, es, z, row, col0);
        }
      } else if (MODE == kUe8m0) {
        // scales already applied by the MMA: all 128 columns into registers,
        // the single accumulator released at once, then the epilogue
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&acc_full[0]), aphase, lim, abort_flag));
        if (!ok) break;
        tc_fence_after();
        const uint32_t taddr = tmem_base + t_row + static_cast<uint32_t>(half * CHUNK);
        float zf[CHUNK];
#pragma unroll
        for (int c = 0; c < CHUNK / 32; ++c)
          tmem_ld_32x32b_x32(taddr + c * 32, *reinterpret_cast<float(*)[32]>(zf + c * 32));
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&acc_empty[0]));
        aphase ^= 1;
        if (EPI == kEpiDenseFp8) {
          ok = dense_fp8_epilogue(p, es, zf, row, col0, m_blk, rit, half, quarter, lane, tcount, blk_bar, blk_max,
                                  lim, abort_flag);
          if (!ok) break;
        } else {
          epi_consume128<EPI>(p, es, zf, row, col0);
        }
      } else if (EPI == kEpiDenseFp8) {
        // tensor / row scaling: all 128 scaled columns into registers, buffer
        // released, then the quantised dense epilogue
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&acc_full[ab]), aphase, lim, abort_flag));
        if (!ok) break;
        tc_fence_after();
        const uint32_t taddr = tmem_base + t_row + static_cast<uint32_t>(ab * BN + half * CHUNK);
        const float sa = (MODE == kTensor) ? __ldg(p.a_scales) : (row_ok ? __ldg(p.a_scales + row) : 0.f);
        float zf[CHUNK];
#pragma unroll
        for (int c = 0; c < CHUNK / 32; ++c) {
          float(&v)[32] = *reinterpret_cast<float(*)[32]>(zf + c * 32);
          tmem_ld_32x32b_x32(taddr + c * 32, v);
          if (MODE == kRow) {
            const int colq = col0 + c * 32 + lane;
            const float sbl = colq < p.N ? __ldg(p.b_scales + colq) : 0.f;
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] *= sa * __shfl_sync(0xffffffffu, sbl, i);
          } else {
            const float s0 = sa * __ldg(p.b_scales);
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] *= s0;
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&acc_empty[ab]));
        ab ^= 1;
        if (ab == 0) aphase ^= 1;
        ok = dense_fp8_epilogue(p, es, zf, row, col0, m_blk, rit, half, quarter, lane, tcount, blk_bar, blk_max,
                                lim, abort_flag);
        if (!ok) break;
      } else {
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&acc_full[ab]), aphase, lim, abort_flag));
        if (!ok) break;
        tc_fence_after();
        const uint32_t taddr = tmem_base + t_row + static_cast<uint32_t>(ab * BN + half * CHUNK);
        const float sa = (MODE == kBf16) ? 1.f
                         : (MODE == kTensor) ? __ldg(p.a_scales)
                                             : (row_ok ? __ldg(p.a_scales + row) : 0.f);
        const float s0 = (MODE == kTensor) ? sa * __ldg(p.b_scales) : 0.f;
#pragma unroll 1
        for (int c = 0; c < CHUNK / 32; ++c) {
          float v[32];
          tmem_ld_32x32b_x32(taddr + c * 32, v);
          if (MODE == kRow) {
            // lane i fetches the scale of column i of this piece; broadcast by shuffle
            const int colq = col0 + c * 32 + lane;
            const float sbl = colq < p.N ? __ldg(p.b_scales + colq) : 0.f;
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] *= sa * __shfl_sync(0xffffffffu, sbl, i);
          } else if (MODE == kTensor) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] *= s0;
          }
          epi_consume32<EPI>(p, es, v, row, col0, c * 32);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&acc_empty[ab]));
        ab ^= 1;
        if (ab == 0) aphase ^= 1;
      }
      epi_finish<EPI>(p, es, row, chunk);
    }
    if (!ok) {
      *abort_flag = 1;
      flag(kErrTimeout);
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ------------------------------------------------------------------ ratios
__global__ void ratios_kernel(const float* __restrict__ a, const float* __restrict__ b, int64_t T,
                              float* __restrict__ r) {
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < T;
       t += (int64_t)gridDim.x * blockDim.x)
    r[t] = expf(a[t] - b[t]);
}

// E8M0 scale-factor images of the UE8M0 mode (layout at SF_IMG_BYTES) from
// the power-of-two float32 scales: activations [num_kb][M] (1x128 blocks),
// weights [n_chunks][num_kb] (128x128 blocks).  One warp per image group:
// first the num_m x num_kg groups of A, then the num_n x num_kg of B.  Rows
// past M or N and K blocks past num_kb get scale 1 (byte 127).
__global__ void ue8m0_pack_kernel(const float* __restrict__ a_scales, const float* __restrict__ b_scales,
                                  int M, int num_kb, int n_chunks, int num_m, int num_n, int num_kg,
                                  uint8_t* __restrict__ sf_a, uint8_t* __restrict__ sf_b) {
  const int64_t w = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t na = static_cast<int64_t>(num_m) * num_kg, nb = static_cast<int64_t>(num_n) * num_kg;
  if (w < na) {
    const int m_blk = static_cast<int>(w / num_kg), g = static_cast<int>(w % num_kg);
    uint32_t word[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int row = m_blk * BM + j * 32 + lane;
      uint32_t v = 0;
#pragma unroll
      for (int q = 0; q < SF_KB; ++q) {
        const int kb = g * SF_KB + q;
        const float sc = (row < M && kb < num_kb) ? a_scales[static_cast<size_t>(kb) * M + row] : 1.f;
        v |= e8m0_byte(sc) << (8 * q);
      }
      word[j] = v;
    }
    reinterpret_cast<uint4*>(sf_a + w * SF_IMG_BYTES)[lane] = make_uint4(word[0], word[1], word[2], word[3]);
  } else if (w < na + nb) {
    const int64_t wb = w - na;
    const int n_blk = static_cast<int>(wb / num_kg), g = static_cast<int>(wb % num_kg);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int chunk = 2 * n_blk + h;
      uint32_t v = 0;
#pragma unroll
      for (int q = 0; q < SF_KB; ++q) {
        const int kb = g * SF_KB + q;
        const float sc = (chunk < n_chunks && kb < num_kb) ? b_scales[static_cast<size_t>(chunk) * num_kb + kb] : 1.f;
        v |= e8m0_byte(sc) << (8 * q);
      }
      reinterpret_cast<uint4*>(sf_b + (wb * 2 + h) * SF_IMG_BYTES)[lane] = make_uint4(v, v, v, v);
    }
  }
}

// Rows selected for dense dlogits are gathered (codes, scales, targets, lse,
// grad) into a contiguous operand for the same GEMM kernel.
__global__ void gather_rows_kernel(const uint8_t* __restrict__ h_codes,
                                   const float* __restrict__ h_scales, int gran, int64_t T,
                                   int64_t H, const int32_t* __restrict__ targets,
                                   const float* __restrict__ lse, const float* __restrict__ grad,
                                   const int64_t* __restrict__ rows, int64_t n_rows,
                                   uint8_t* __restrict__ g_codes, float* __restrict__ g_scales,
                                   int32_t* __restrict__ g_targets, float* __restrict__ g_lse,
                                   float* __restrict__ g_grad) {
  const int64_t i = blockIdx.x;
  if (i >= n_rows) return;
  int64_t t = rows[i];
  const bool ok = t >= 0 && t < T;
  if (!ok) {
    if (threadIdx.x == 0) flag(kErrDevice);
    t = 0;
  }
  const uint4* src = reinterpret_cast<const uint4*>(h_codes + t * H);
  uint4* dst = reinterpret_cast<uint4*>(g_codes + i * H);
  for (int64_t v = threadIdx.x; v < H / 16; v += blockDim.x) dst[v] = ok ? src[v] : make_uint4(0, 0, 0, 0);
  if (threadIdx.x == 0) {
    g_targets[i] = targets[t];
    g_lse[i] = lse[t];
    g_grad[i] = ok ? grad[t] : NAN;
    if (gran == kTensor) {
      if (i == 0) g_scales[0] = h_scales[0];
    } else if (gran == kRow) {
      g_scales[i] = h_scales[t];
    }
  }
  if (gran == kBlock || gran == kUe8m0) {
    const int64_t nkb = H / 128;
    for (int64_t kb = threadIdx.x; kb < nkb; kb += blockDim.x) g_scales[kb * n_rows + i] = h_scales[kb * T + t];
  }
}

__global__ void wait_selftest_kernel(uint64_t limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    fence_mbar_init();
    // nothing ever arrives on this barrier: the wait must expire
    if (!mbar_wait(smem_u32(&bar), 0, limit_ns, nullptr)) flag(kErrTimeout);
  }
}

// ------------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

// K-major matrix [rows][K] with row stride `ld` elements, box of 128 bytes
// along K x box_rows, 128B swizzle, zero fill outside the matrix: uint8 E4M3
// codes (128 elements per box row) or bf16 values (64 elements).
bool make_tmap(CUtensorMap* tm, const void* base, int64_t rows, int64_t K, int64_t ld,
               uint32_t box_rows, bool bf16) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  const int esize = bf16 ? 2 : 1;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld * esize)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK / esize), box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(tm, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8, 2,
                  const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int MODE, int EPI>
cudaError_t launch_mode(const CUtensorMap& ta, const CUtensorMap& tb, const Params& p, int grid,
                        cudaStream_t s) {
  auto kern = fp8_gemm_kernel<MODE, EPI>;
  static int configured_device = -1;
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured_device != dev) {
    // The warpgroups re-split the registers the CTA was launched with
    // (setmaxnreg): each SM sub-partition holds one control warp and two
    // epilogue warps, so 3 x (launch registers) must cover 56 + 2 x 224.
    // Refuse to launch a build where that does not hold (it would wait forever).
    cudaFuncAttributes attr;
    cudaError_t e = cudaFuncGetAttributes(&attr, kern);
    if (e != cudaSuccess) return e;
    if (attr.numRegs * 3 < CTRL_REGS + 2 * EPI_REGS ||
        attr.numRegs * THREADS < 128 * CTRL_REGS + EPI_WARPS * 32 * EPI_REGS)
      return cudaErrorInvalidConfiguration;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem_bytes<MODE>()));
    if (e != cudaSuccess) return e;
    configured_device = dev;
  }
  kern<<<grid, THREADS, smem_bytes<MODE>(), s>>>(ta, tb, p);
  return cudaGetLastError();
}

template <int EPI>
cudaError_t launch_gemm(const GemmArgs& a, cudaStream_t s) {
  if (a.M == 0 || a.N == 0) return cudaSuccess;
  const bool bf16 = a.gran == kBf16;
  CUtensorMap ta, tb;
  if (!make_tmap(&ta, a.a_codes, a.M, a.K, a.lda ? a.lda : a.K, BM, bf16) ||
      !make_tmap(&tb, a.b_codes, a.N, a.K, a.ldb ? a.ldb : a.K, BN, bf16))
    return cudaErrorInvalidValue;
  Params p{};
  p.a_scales = a.a_scales;
  p.b_scales = a.b_scales;
  p.targets = a.targets;
  p.partials = a.partials;
  p.zy = a.zy;
  p.lse = a.lse;
  p.grad = a.grad;
  p.out = a.out;
  p.pq_out = a.pq_out;
  p.pq_scales = a.pq_scales;
  p.ptq_out = a.ptq_out;
  p.ptq_scales = a.ptq_scales;
  p.ld_pq = a.ld_pq;
  p.ld_ptq = a.ld_ptq;
  p.c_out = a.c_out;
  p.ld_c = a.ld_c;
  p.accumulate = a.accumulate;
  p.p_pow2 = a.p_pow2;
  p.M = static_cast<int>(a.M);
  p.N = static_cast<int>(a.N);
  p.K = static_cast<int>(a.K);
  p.num_m = static_cast<int>((a.M + BM - 1) / BM);
  p.num_n = static_cast<int>((a.N + BN - 1) / BN);
  p.band_m = EPI == kEpiStore ? kBandStore : kBandM;
  const int64_t bk_elems = bf16 ? BK / 2 : BK;  // K elements per 128-byte stage row
  p.num_kb = static_cast<int>((a.K + bk_elems - 1) / bk_elems);
  p.n_chunks = static_cast<int>((a.N + CHUNK - 1) / CHUNK);
  p.wait_limit_ns = wait_limit_ns();
  if (a.gran == kUe8m0) {
    if (a.sf_images == nullptr || (reinterpret_cast<uintptr_t>(a.sf_images) & 15u) != 0)
      return cudaErrorInvalidValue;
    p.num_kg = (p.num_kb + SF_KB - 1) / SF_KB;
    uint8_t* sf_a = a.sf_images;
    uint8_t* sf_b = sf_a + static_cast<size_t>(p.num_m) * p.num_kg * SF_IMG_BYTES;
    p.sf_a = sf_a;
    p.sf_b = sf_b;
    const int64_t warps = (static_cast<int64_t>(p.num_m) + p.num_n) * p.num_kg;
    ue8m0_pack_kernel<<<static_cast<unsigned>((warps + 7) / 8), 256, 0, s>>>(
        a.a_scales, a.b_scales, p.M, p.num_kb, p.n_chunks, p.num_m, p.num_n, p.num_kg, sf_a, sf_b);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  const int64_t tiles = static_cast<int64_t>(p.num_m) * p.num_n;
  const int grid = static_cast<int>(tiles < sm_count() ? tiles : sm_count());
  if constexpr (EPI == kEpiStore) {  // plain fp32 store: block-scaled FP8 (backward, both scale formats) or BF16
    switch (a.gran) {
      case kBlock: return launch_mode<kBlock, EPI>(ta, tb, p, grid, s);
      case kUe8m0: return launch_mode<kUe8m0, EPI>(ta, tb, p, grid, s);
      case kBf16: return launch_mode<kBf16, EPI>(ta, tb, p, grid, s);
      default: return cudaErrorInvalidValue;
    }
  } else if constexpr (EPI == kEpiDenseFp8) {  // recomputed FP8 logits only
    switch (a.gran) {
      case kTensor: return launch_mode<kTensor, EPI>(ta, tb, p, grid, s);
      case kRow: return launch_mode<kRow, EPI>(ta, tb, p, grid, s);
      case kBlock: return launch_mode<kBlock, EPI>(ta, tb, p, grid, s);
      case kUe8m0: return launch_mode<kUe8m0, EPI>(ta, tb, p, grid, s);
      default: return cudaErrorInvalidValue;
    }
  } else {
    switch (a.gran) {
      case kTensor: return launch_mode<kTensor, EPI>(ta, tb, p, grid, s);
      case kRow: return launch_mode<kRow, EPI>(ta, tb, p, grid, s);
      case kBf16: return launch_mode<kBf16, EPI>(ta, tb, p, grid, s);
      case kUe8m0: return launch_mode<kUe8m0, EPI>(ta, tb, p, grid, s);
      default: return launch_mode<kBlock, EPI>(ta, tb, p, grid, s);
    }
  }
}

int blocks_for(int64_t n, int threads) {
  int64_t b = (n + threads - 1) / threads;
  return static_cast<int>(b < 1 ? 1 : b);
}

}  // namespace

int64_t gemm_partials_per_token(int64_t N) { return (N + CHUNK - 1) / CHUNK; }

size_t gemm_ue8m0_image_bytes(int64_t M, int64_t N, int64_t K) {
  if (M < 1 || N < 1 || K < 1) return 0;
  const int64_t num_m = (M + BM - 1) / BM, num_n = (N + BN - 1) / BN;
  const int64_t num_kg = ((K + BK - 1) / BK + SF_KB - 1) / SF_KB;
  return align_up(static_cast<size_t>((num_m + 2 * num_n) * num_kg) * SF_IMG_BYTES, 256);
}

cudaError_t launch_gemm_lse(const GemmArgs& a, cudaStream_t s) { return launch_gemm<kEpiLse>(a, s); }

cudaError_t launch_gemm_dlogits(const GemmArgs& a, cudaStream_t s) {
  return launch_gemm<kEpiDlogits>(a, s);
}

cudaError_t launch_gemm_dense_dlogits(const GemmArgs& a, cudaStream_t s) {
  return launch_gemm<kEpiDenseFp8>(a, s);
}

cudaError_t launch_gemm_store(const GemmArgs& a, cudaStream_t s) { return launch_gemm<kEpiStore>(a, s); }

cudaError_t launch_ratios(const float* lp_new, const float* lp_old, int64_t T, float* r,
                          cudaStream_t s) {
  if (T == 0) return cudaSuccess;
  int b = blocks_for(T, 256);
  if (b > sm_count() * 8) b = sm_count() * 8;
  ratios_kernel<<<b, 256, 0, s>>>(lp_new, lp_old, T, r);
  return cudaGetLastError();
}

cudaError_t launch_gather_rows(const uint8_t* h_codes, const float* h_scales, int gran, int64_t T,
                               int64_t H, const int32_t* targets, const float* lse,
                               const float* grad, const int64_t* rows, int64_t n_rows,
                               uint8_t* g_codes, float* g_scales, int32_t* g_targets,
                               float* g_lse, float* g_grad, cudaStream_t s) {
  if (n_rows == 0) return cudaSuccess;
  gather_rows_kernel<<<static_cast<unsigned>(n_rows), 128, 0, s>>>(
      h_codes, h_scales, gran, T, H, targets, lse, grad, rows, n_rows, g_codes, g_scales,
      g_targets, g_lse, g_grad);
  return cudaGetLastError();
}

cudaError_t launch_wait_selftest(uint64_t limit_ns, cudaStream_t s) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(limit_ns);
  return cudaGetLastError();
}

uint32_t gemm_status_take() {
  uint32_t v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, d_status, sizeof(v)) != cudaSuccess) return 0;
  cudaMemcpyToSymbol(d_status, &z, sizeof(z));
  return v;
}

}  // namespace fp8rl
