// a3 in block scaling (Eq. 3 with 1x128 activation and 128x128 weight
// blocks, §2.2) on CTA pairs: the FP8 lm_head GEMM whose epilogue promotes
// every 128-wide K block, acc += S_h[t][kb] S_W[vb][kb] * partial, then streams
// the logsumexp and the target gather (the epilogues are those of gemm.cu).
//
// Why a pair: the promotion needs each K block's partial product in its own
// TMEM buffer, and one CTA's 512 TMEM columns hold only two 128 x 256
// buffers, so the MMA of K block kb + 2 waits for the epilogue to have read
// kb -- a latency chain longer than one K block of MMA work.  A cluster of two
// CTAs on two SMs shares one 256 (tokens) x 128 (vocabulary) tile:
// tcgen05.mma.cta_group::2 reads 128 token rows of A from each CTA's shared
// memory and 64 vocabulary rows of B from each, and writes each CTA's 128 x 128
// accumulator into its own TMEM.  With 128 columns per buffer every SM holds
// four buffers (three K blocks of slack), at the same shared-memory operand
// bytes per FLOP as a 128 x 256 tile on one SM.
//
// Roles (12 warps per CTA, both CTAs):
//   warp 0      TMA producer of this CTA's A (128 x 128 B) and B (64 x 128 B)
//               boxes into an 8-stage ring; completions land on its own
//               full barrier;
//   warp 1      even CTA: MMA issuer (M = 256, N = 128, K = 32 per
//               instruction, four per K block), commits multicast to both
//               CTAs' empty / accumulator-full barriers; odd CTA: idle;
//   warp 2      scale loader: this CTA's 128 activation scales and the tile's
//               weight scale of four K blocks per ring slot;
//   warp 3      odd CTA: forwards each landed stage to the even CTA's full
//               barrier (so the MMA issues only once both halves are in);
//               even CTA: idle;
//   warps 4..11 epilogue: one thread per token row and 64 vocabulary columns;
//               buffer release arrives on the even CTA's accumulator-empty
//               barrier (both CTAs' epilogues must have read it).
// Every wait is bounded; a cluster barrier before exit keeps each CTA alive
// while its partner may still touch its shared memory or TMEM.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "gemm_epi.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

__device__ uint32_t d_status;

__device__ __forceinline__ void flag(uint32_t bits) { atomicOr(&d_status, bits); }

constexpr int PM = 256;            // tokens per pair tile (128 per CTA = TMEM lanes)
constexpr int PN = 128;            // vocabulary columns per pair tile (64 B rows per CTA)
constexpr int CM = 128;            // token rows per CTA
constexpr int CN = 64;             // B rows per CTA
constexpr int BK = 128;            // K bytes per stage (one K block of 128 E4M3 codes)
constexpr int STAGES = 8;
constexpr int NBUF = 4;            // TMEM accumulator buffers of PN columns
constexpr int EPI_WARPS = 8;
constexpr int EPI_WARP0 = 4;
constexpr int THREADS = 128 + EPI_WARPS * 32;
constexpr int CTRL_REGS = 56;
constexpr int EPI_REGS = 224;
constexpr uint32_t A_BYTES = CM * BK;
constexpr uint32_t B_BYTES = CN * BK;
constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
constexpr uint32_t TMEM_COLS = NBUF * PN;
constexpr int SC_SLOTS = 4;
constexpr int SC_KB = 4;
constexpr uint32_t SC_KB_FLOATS = CM + 4;  // 128 activation + 1 weight (+3 pad)
constexpr uint32_t SC_SLOT_FLOATS = SC_KB * SC_KB_FLOATS;
constexpr uint32_t SC_BYTES = SC_SLOTS * SC_SLOT_FLOATS * 4;
// Merge slots of the LSE epilogue's two column halves: a half can run at most
// NBUF tiles ahead of the other (it cannot pass a K block whose buffer the
// other half has not released), so 8 slots are never reused too early.
constexpr int MERGE_SLOTS = 8;
constexpr uint32_t MERGE_BYTES = MERGE_SLOTS * 4 * 32 * 16;  // slots x lane quarters x lanes x float4
constexpr size_t SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + SC_BYTES + MERGE_BYTES + 1024;
constexpr uint64_t kDrainNs = 1000000000ull;
constexpr int kBandPairs = 32;     // pair tiles per band of the tile order (8192 tokens)

template <int EPI>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
    fp8_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                         const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* smA = smem;
  uint8_t* smB = smem + STAGES * A_BYTES;
  float* sc_ring = reinterpret_cast<float*>(smB + STAGES * B_BYTES);
  float4* merge = reinterpret_cast<float4*>(reinterpret_cast<uint8_t*>(sc_ring) + SC_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(merge) + MERGE_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = full + STAGES;
  uint64_t* acc_full = empty + STAGES;
  uint64_t* acc_empty = acc_full + NBUF;
  uint64_t* sc_full = acc_empty + NBUF;
  uint64_t* sc_empty = sc_full + SC_SLOTS;
  uint64_t* done = sc_empty + SC_SLOTS;
  uint64_t* merged = done + 1;  // [MERGE_SLOTS][4]: second half's values written
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(merged + MERGE_SLOTS * 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      // the even CTA's stage is full once its own copies landed (arrive +
      // bytes) and the odd CTA forwarded that its half landed too
      mbar_init(smem_u32(&full[s]), leader ? 2 : 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int b = 0; b < NBUF; ++b) {
      mbar_init(smem_u32(&acc_full[b]), 1);
      mbar_init(smem_u32(&acc_empty[b]), 2 * EPI_WARPS);
    }
    for (int i = 0; i < SC_SLOTS; ++i) {
      mbar_init(smem_u32(&sc_full[i]), 32);
      mbar_init(smem_u32(&sc_empty[i]), EPI_WARPS);
    }
    mbar_init(smem_u32(done), 1);
    for (int i = 0; i < MERGE_SLOTS * 4; ++i) mbar_init(smem_u32(&merged[i]), 32);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(tmem_holder), TMEM_COLS);
    tmem_relinquish_pair();
  }
  // barrier initialisation and the TMEM allocation become visible to both CTAs
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
  const int total = p.num_m * p.num_n;
  const uint64_t lim = p.wait_limit_ns;

  if (warp < EPI_WARP0) {
    warpgroup_reg_dealloc<CTRL_REGS>();
    if (warp == 0) {
      // ---------------------------------------------------------- producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_phase = 0;
      bool ok = true;
      for (int tile = pair; tile < total && ok; tile += n_pairs) {
        int m_blk, n_blk;
        tile_coords(tile, p, m_blk, n_blk);
        const int m0 = m_blk * PM + static_cast<int>(rank) * CM;
        const int n0 = n_blk * PN + static_cast<int>(rank) * CN;
        for (int kb = 0; kb < p.num_kb; ++kb) {
          ok = __all_sync(0xffffffffu, mbar_wait_cluster(smem_u32(&empty[stage]), phase ^ 1, lim, abort_flag));
          if (!ok) break;
          if (elect_one()) {
            mbar_arrive_expect_tx(smem_u32(&full[stage]), STAGE_BYTES);
            tma_load_2d(smem_u32(smA + stage * A_BYTES), &tmA, smem_u32(&full[stage]), kb * BK, m0);
            tma_load_2d(smem_u32(smB + stage * B_BYTES), &tmB, smem_u32(&full[stage]), kb * BK, n0);
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
      // no copy in flight, and every MMA commit for these stages landed, before exit
      for (int s = 0; s < STAGES; ++s)
        if (armed & (1u << s)) {
          const uint32_t ph = (armed_phase >> s) & 1;
          mbar_wait(smem_u32(&full[s]), ph, kDrainNs, nullptr);
          if (ok) mbar_wait_cluster(smem_u32(&empty[s]), ph, kDrainNs, nullptr);
        }
    } else if (warp == 1 && leader) {
      // ---------------------------------------------------------- MMA issuer
      int stage = 0, ab = 0;
      uint32_t phase = 0, aphase = 0;
      constexpr uint32_t idesc = idesc_e4m3_f32(PM, PN);
      bool ok = true;
      for (int tile = pair; tile < total && ok; tile += n_pairs) {
        for (int kb = 0; kb < p.num_kb; ++kb) {
          ok = __all_sync(0xffffffffu, mbar_wait_cluster(smem_u32(&full[stage]), phase, lim, abort_flag));
          if (!ok) break;
          ok = __all_sync(0xffffffffu, mbar_wait_cluster(smem_u32(&acc_empty[ab]), aphase ^ 1, lim, abort_flag));
          if (!ok) break;
          tc_fence_after();
          const uint32_t d = tmem_base + static_cast<uint32_t>(ab * PN);
          const uint64_t adesc = smem_desc_sw128(smem_u32(smA + stage * A_BYTES));
          const uint64_t bdesc = smem_desc_sw128(smem_u32(smB + stage * B_BYTES));
#pragma unroll
          for (int k = 0; k < BK / 32; ++k)  // +32 bytes along K inside the swizzled row
            mma_f8f6f4_pair_elect(d, adesc + 2 * k, bdesc + 2 * k, idesc, k > 0);
          mma_commit_pair_elect(smem_u32(&empty[stage]), 0x3);
          mma_commit_pair_elect(smem_u32(&acc_full[ab]), 0x3);
          if (++ab == NBUF) {
            ab = 0;
            aphase ^= 1;
          }
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
      mma_commit_pair_elect(smem_u32(done), 0x1);
      mbar_wait(smem_u32(done), 0, kDrainNs, nullptr);
    } else if (warp == 2) {
      // ---------------------------------------------------------- scale loader
      int slot = 0;
      uint32_t sphase = 0;
      bool ok = true;
      for (int tile = pair; tile < total && ok; tile += n_pairs) {
        int m_blk, n_blk;
        tile_coords(tile, p, m_blk, n_blk);
        const int m0 = m_blk * PM + static_cast<int>(rank) * CM;
        for (int kg = 0; kg < p.num_kb; kg += SC_KB) {
          ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&sc_empty[slot]), sphase ^ 1, lim, abort_flag));
          if (!ok) break;
          const int nkb = min(SC_KB, p.num_kb - kg);
          for (int q = 0; q < nkb; ++q) {
            const int kb = kg + q;
            const uint32_t dst = smem_u32(sc_ring + slot * SC_SLOT_FLOATS + q * SC_KB_FLOATS);
            const float* src = p.a_scales + static_cast<size_t>(kb) * p.M;
#pragma unroll
            for (int j = 0; j < CM / 32; ++j) {
              const int r = m0 + j * 32 + lane;
              if (r < p.M) cp_async_4(dst + (j * 32 + lane) * 4, src + r);
            }
            if (lane == 0) cp_async_4(dst + CM * 4, p.b_scales + static_cast<size_t>(n_blk) * p.num_kb + kb);
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
      asm volatile("cp.async.wait_all;" ::: "memory");
    } else if (warp == 3 && !leader) {
      // ---------------------------------------------------------- forwarder
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int tile = pair; tile < total && ok; tile += n_pairs) {
        for (int kb = 0; kb < p.num_kb; ++kb) {
          ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&full[stage]), phase, lim, abort_flag));
          if (!ok) break;
          if (lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(&full[stage]), 0));
          __syncwarp();
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
    }
  } else {
    warpgroup_reg_alloc<EPI_REGS>();
    // ------------------------------------------------------------ epilogue
    const int ew = warp - EPI_WARP0;
    const int quarter = warp & 3;  // TMEM lanes this warp may access
    const int half = ew >> 2;      // which 64 columns of the 128-wide tile
    const int rit = quarter * 32 + lane;
    const uint32_t t_row = static_cast<uint32_t>(quarter * 32) << 16;
    int ab = 0, sslot = 0, tcount = 0;
    uint32_t aphase = 0, sphase = 0;
    bool ok = true;
    for (int tile = pair; tile < total && ok; tile += n_pairs, ++tcount) {
      int m_blk, n_blk;
      tile_coords(tile, p, m_blk, n_blk);
      const int row = m_blk * PM + static_cast<int>(rank) * CM + rit;
      const int col0 = n_blk * PN + half * (PN / 2);
      EpiState es;
      epi_begin<EPI>(p, es, row, col0);
      float2 z2[PN / 4];
#pragma unroll
      for (int i = 0; i < PN / 4; ++i) z2[i] = make_float2(0.f, 0.f);
      for (int kb = 0; kb < p.num_kb; ++kb) {
        const int q = kb % SC_KB;
        if (q == 0) {
          ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&sc_full[sslot]), sphase, lim, abort_flag));
          if (!ok) break;
        }
        const float* scs = sc_ring + sslot * SC_SLOT_FLOATS + q * SC_KB_FLOATS;
        const float sc = scs[rit] * scs[CM];
        if (q == SC_KB - 1 || kb == p.num_kb - 1) {
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&sc_empty[sslot]));
          if (++sslot == SC_SLOTS) {
            sslot = 0;
            sphase ^= 1;
          }
        }
        ok = __all_sync(0xffffffffu, mbar_wait_cluster(smem_u32(&acc_full[ab]), aphase, lim, abort_flag));
        if (!ok) break;
        tc_fence_after();
        const uint32_t taddr = tmem_base + t_row + static_cast<uint32_t>(ab * PN + half * (PN / 2));
        uint32_t ra[32], rb[32];
        tmem_ld_32x32b_x32_issue(taddr, ra);
        tmem_ld_32x32b_x32_issue(taddr + 32, rb);
        tmem_wait_ld(ra);
        tmem_wait_ld(rb);
        // both pieces are in registers: hand the buffer back to the MMA
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(&acc_empty[ab]), 0));
#pragma unroll
        for (int i = 0; i < 16; ++i)
          ffma2(z2[i].x, z2[i].y, __uint_as_float(ra[2 * i]), __uint_as_float(ra[2 * i + 1]), sc);
#pragma unroll
        for (int i = 0; i < 16; ++i)
          ffma2(z2[16 + i].x, z2[16 + i].y, __uint_as_float(rb[2 * i]), __uint_as_float(rb[2 * i + 1]), sc);
        if (++ab == NBUF) {
          ab = 0;
          aphase ^= 1;
        }
      }
      if (!ok) break;
      const float* z = reinterpret_cast<const float*>(z2);
      epi_consume32<EPI>(p, es, z, row, col0, 0);
      epi_consume32<EPI>(p, es, z + 32, row, col0, 32);
      if (EPI == kEpiLse) {
        // the two 64-column halves of a row meet in shared memory: the second
        // half writes its (max, sum exp, z_y) and arrives; the first half
        // waits (bounded), merges and writes the chunk's one partial
        const int ms = tcount % MERGE_SLOTS;
        const uint32_t mpar = static_cast<uint32_t>(tcount / MERGE_SLOTS) & 1u;
        float4* slot = merge + (ms * 4 + quarter) * 32 + lane;
        const uint32_t mbar = smem_u32(&merged[ms * 4 + quarter]);
        const bool has_y = es.j >= 0 && es.j < PN / 2;
        if (half == 1) {
          *slot = make_float4(es.m, es.s, es.zy, has_y ? 1.f : 0.f);
          mbar_arrive(mbar);
        } else {
          ok = __all_sync(0xffffffffu, mbar_wait(mbar, mpar, lim, abort_flag));
          if (!ok) break;
          if (row < p.M && n_blk < p.n_chunks) {
            const float4 o = *slot;
            float m = es.m, sum = es.s;
            if (o.x != -INFINITY) {
              const float mn = fmaxf(m, o.x);
              sum = sum * exp2f((m - mn) * kLog2e) + o.y * exp2f((o.x - mn) * kLog2e);
              m = mn;
            }
            p.partials[static_cast<size_t>(n_blk) * p.M + row] = make_float2(m, sum);
            if (has_y) p.zy[row] = es.zy;
            else if (o.w != 0.f) p.zy[row] = o.z;
          }
        }
      }
    }
    if (!ok) {
      *abort_flag = 1;
      flag(kErrTimeout);
    }
    tc_fence_before();
  }
  __syncthreads();
  // neither CTA leaves while the other may still read its shared memory
  // (the pair MMA), arrive on its barriers or hold the shared TMEM
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, TMEM_COLS);
  }
}

// K-major E4M3 matrix [rows][K] (row stride `ld` bytes), box of 128 bytes along
// K x box_rows, 128-byte swizzle, zero fill outside the matrix.
bool make_tmap_e4m3(CUtensorMap* tm, const void* base, int64_t rows, int64_t K, int64_t ld, uint32_t box_rows) {
  auto fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(tensormap_encoder());
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(tm, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct DevCfg {
  int device = -1;
  int max_clusters = 0;
};

template <int EPI>
cudaError_t launch_pair(const CUtensorMap& ta, const CUtensorMap& tb, const Params& p, cudaStream_t s) {
  auto kern = fp8_gemm_pair_kernel<EPI>;
  static DevCfg cfg;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (cfg.device != dev) {
    // setmaxnreg re-splits the registers the CTA was launched with: each SM
    // sub-partition holds one control warp and two epilogue warps, so
    // 3 x (launch registers) must cover 56 + 2 x 224.  Refuse a build where
    // that does not hold (it would wait forever).
    cudaFuncAttributes attr;
    e = cudaFuncGetAttributes(&attr, kern);
    if (e != cudaSuccess) return e;
    if (attr.numRegs * 3 < CTRL_REGS + 2 * EPI_REGS ||
        attr.numRegs * THREADS < 128 * CTRL_REGS + EPI_WARPS * 32 * EPI_REGS)
      return cudaErrorInvalidConfiguration;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(SMEM_BYTES));
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t lc = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.gridDim = dim3(2 * static_cast<unsigned>(sm_count()));
    lc.blockDim = dim3(THREADS);
    lc.dynamicSmemBytes = SMEM_BYTES;
    lc.attrs = at;
    lc.numAttrs = 1;
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, kern, &lc);
    if (e != cudaSuccess) return e;
    if (n < 1) return cudaErrorInvalidConfiguration;
    cfg.max_clusters = n;
    cfg.device = dev;
  }
  const int64_t tiles = static_cast<int64_t>(p.num_m) * p.num_n;
  const int pairs = static_cast<int>(tiles < cfg.max_clusters ? tiles : cfg.max_clusters);
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(2 * static_cast<unsigned>(pairs));
  lc.blockDim = dim3(THREADS);
  lc.dynamicSmemBytes = SMEM_BYTES;
  lc.stream = s;
  // the cluster shape is compiled in (__cluster_dims__)
  return cudaLaunchKernelEx(&lc, kern, ta, tb, p);
}

}  // namespace

cudaError_t launch_gemm_pair(const GemmArgs& a, int epi, cudaStream_t s) {
  if (a.M == 0 || a.N == 0) return cudaSuccess;
  if (a.gran != FP8RL_GRAN_BLOCK || a.K % BK != 0) return cudaErrorInvalidValue;
  CUtensorMap ta, tb;
  if (!make_tmap_e4m3(&ta, a.a_codes, a.M, a.K, a.lda ? a.lda : a.K, CM) ||
      !make_tmap_e4m3(&tb, a.b_codes, a.N, a.K, a.ldb ? a.ldb : a.K, CN))
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
  p.p_out = a.p_out;
  p.pt_out = a.pt_out;
  p.ld_p = a.ld_p;
  p.ld_pt = a.ld_pt;
  p.M = static_cast<int>(a.M);
  p.N = static_cast<int>(a.N);
  p.K = static_cast<int>(a.K);
  p.num_m = static_cast<int>((a.M + PM - 1) / PM);
  p.num_n = static_cast<int>((a.N + PN - 1) / PN);
  p.band_m = kBandPairs;
  p.num_kb = static_cast<int>(a.K / BK);
  p.n_chunks = static_cast<int>((a.N + CHUNK - 1) / CHUNK);
  p.wait_limit_ns = wait_limit_ns();
  switch (epi) {
    case kEpiLse: return launch_pair<kEpiLse>(ta, tb, p, s);
    case kEpiDlogits: return launch_pair<kEpiDlogits>(ta, tb, p, s);
    case kEpiDense: return launch_pair<kEpiDense>(ta, tb, p, s);
    default: return cudaErrorInvalidValue;
  }
}

uint32_t gemm_pair_status_take() {
  uint32_t v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, d_status, sizeof(v)) != cudaSuccess) return 0;
  cudaMemcpyToSymbol(d_status, &z, sizeof(z));
  return v;
}

}  // namespace fp8rl
