// bf16 GEMM on the 5th-generation tensor cores (tcgen05 + TMEM), operands staged
// by TMA, for every dense contraction of the path: the selector encoder, the
// projector and the LM prefill (QKV with fused RoPE, O + residual, gate/up with
// fused SwiGLU, down + residual).
//
// C[M, N] = A[M, K] * B[N, K]^T: A row-major activations, B an nn.Linear weight.
// Persistent kernel, one CTA per SM, 6 warps:
//   warp 0      TMA producer: A tile 128x64 and B tile BNx64 per stage (128-byte
//               swizzle), STAGES-deep ring guarded by full/empty mbarriers;
//   warp 1      allocates 2*BN TMEM columns (double-buffered fp32 accumulators)
//               and one lane issues tcgen05.mma (M=128, N=BN, K=16) per 16-wide
//               K slice, committing each stage back to the producer;
//   warps 2-5   epilogue: tcgen05.ld of the accumulator (warp w reads TMEM lanes
//               32*(w%4)..+31 = tile rows), fused epilogue math, global stores,
//               then release the accumulator buffer.
// The epilogue of tile i overlaps the main loop of tile i+1.  Every mbarrier
// wait is bounded (SP_DEVERR_TIMEOUT).
//
// A second variant pairs two CTAs on two SMs (cta_group::2, 256-row tiles) so
// each SM stages half of the B tile; it is used wherever M fills a pair tile
// (gemm_pair_policy), the single-CTA kernel elsewhere.
#include <algorithm>
#include <cstdlib>
#include <cstring>

#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

constexpr int BM = 128;
constexpr int BK = 64;

template <int BN>
struct Cfg {
  static constexpr int STAGES = (BN == 256) ? 4 : 6;
  static constexpr uint32_t A_BYTES = BM * BK * 2;
  static constexpr uint32_t B_BYTES = BN * BK * 2;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
  static constexpr size_t SMEM = 1024 + STAGES * (A_BYTES + B_BYTES) + 256;
};

struct KArgs {
  int M_cap;
  const int* M_dev;
  int N_acc;       // accumulator columns over the whole GEMM
  int K;
  GemmEpi e;
  int* err;
};

SP_DEVINL void store_bf16x32(__nv_bfloat16* dst, const float (&v)[32]) {
  uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint4 u;
    u.x = pack_bf16x2(v[8 * q + 0], v[8 * q + 1]);
    u.y = pack_bf16x2(v[8 * q + 2], v[8 * q + 3]);
    u.z = pack_bf16x2(v[8 * q + 4], v[8 * q + 5]);
    u.w = pack_bf16x2(v[8 * q + 6], v[8 * q + 7]);
    d[q] = u;
  }
}

// Drains one 128 x BN accumulator tile from TMEM (this warp: 32 rows, lane =
// row `row`), applies the epilogue and stores the row if it is live.
template <int BN, int EPI>
SP_DEVINL void epilogue_tile(const GemmEpi& e, uint32_t taddr, int row, bool live, int nb, int* err) {
  float v[32];

  if (EPI == EPI_SWIGLU_BF16) {
    float u[32];
#pragma unroll 1
    for (int c = 0; c < BN / 64; ++c) {
      tmem_ld_32x32b_x32(taddr + c * 32, v);
      tmem_ld_32x32b_x32(taddr + BN / 2 + c * 32, u);
      tmem_ld_wait();
      if (live) {
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = silu(v[i]) * u[i];
        __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(e.out) + (size_t)row * e.ldo +
                           nb * (BN / 2) + c * 32;
        store_bf16x32(o, v);
      }
    }
  } else if (EPI == EPI_BF16_ROPE) {
    const int dh = e.head_dim;
    const int half = dh >> 1;
    const int p = live ? __ldg(e.pos + row) : 0;
    const bool pos_ok = p >= 0 && p < e.max_pos;
    if (live && !pos_ok) set_error(err, SP_DEVERR_INDEX);
    float u[32];
#pragma unroll 1
    for (int hb = 0; hb < BN; hb += dh) {
      const int col0 = nb * BN + hb;
      if (col0 < e.rope_cols) {
#pragma unroll 1
        for (int c = 0; c < half; c += 32) {
          tmem_ld_32x32b_x32(taddr + hb + c, v);
          tmem_ld_32x32b_x32(taddr + hb + half + c, u);
          tmem_ld_wait();
          if (live) {
            const float2* cs = e.rope + (size_t)(pos_ok ? p : 0) * half + c;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float2 r = __ldg(cs + i);
              const float a = v[i], b = u[i];
              v[i] = a * r.x - b * r.y;
              u[i] = b * r.x + a * r.y;
            }
            __nv_bfloat16* o =
                reinterpret_cast<__nv_bfloat16*>(e.out) + (size_t)row * e.ldo + col0 + c;
            store_bf16x32(o, v);
            store_bf16x32(o + half, u);
          }
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < dh; c += 32) {
          tmem_ld_32x32b_x32(taddr + hb + c, v);
          tmem_ld_wait();
          if (live) {
            __nv_bfloat16* o =
                reinterpret_cast<__nv_bfloat16*>(e.out) + (size_t)row * e.ldo + col0 + c;
            store_bf16x32(o, v);
          }
        }
      }
    }
  } else {
    int orow = row;
    if (EPI == EPI_SCATTER_BF16 && live) {
      orow = __ldg(e.row_map + row);
      if (orow < 0) {
        set_error(err, SP_DEVERR_INDEX);
      }
    }
    const bool store = live && orow >= 0;
#pragma unroll 1
    for (int c = 0; c < BN / 32; ++c) {
      tmem_ld_32x32b_x32(taddr + c * 32, v);
      tmem_ld_wait();
      if (!store) continue;
      const int col = nb * BN + c * 32;
      if (EPI == EPI_F32 || EPI == EPI_F32_ACC) {
        float4* o = reinterpret_cast<float4*>(reinterpret_cast<float*>(e.out) +
                                              (size_t)orow * e.ldo + col);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          float4 w = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          if (EPI == EPI_F32_ACC) {
            const float4 r = o[q];
            w.x += r.x; w.y += r.y; w.z += r.z; w.w += r.w;
          }
          o[q] = w;
        }
      } else {
        if (EPI == EPI_GELU_BF16) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = gelu_erf(v[i]);
        }
        __nv_bfloat16* o =
            reinterpret_cast<__nv_bfloat16*>(e.out) + (size_t)orow * e.ldo + col;
        store_bf16x32(o, v);
      }
    }
  }
}

template <int BN, int EPI>
__global__ void __launch_bounds__(192, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               const KArgs args) {
  using C = Cfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + C::STAGES * C::B_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tfull = empty + C::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* done = tempty + 2;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(done + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  int* err = args.err;

  int M = args.M_cap;
  if (args.M_dev) M = min(M, __ldg(args.M_dev));
  if (M < 0) M = 0;
  const int num_m = (M + BM - 1) / BM;
  const int num_n = args.N_acc / BN;
  const int total = num_m * num_n;
  const int KB = args.K / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 4);
    }
    mbar_init(done, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tslot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tslot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      int s = 0;
      uint32_t ph = 0;
      int issued = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
        const int mb = t % num_m, nb = t / num_m;
        const int m0 = mb * BM;
        int b0, b1;
        if (EPI == EPI_SWIGLU_BF16) {
          b0 = nb * (BN / 2);
          b1 = args.e.up_off + nb * (BN / 2);
        } else {
          b0 = nb * BN;
          b1 = nb * BN + BN / 2;
        }
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(&empty[s], ph ^ 1u, err)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[s], C::A_BYTES + C::B_BYTES);
          tma_load_2d(sA + s * C::A_BYTES, &tmA, &full[s], kb * BK, m0);
          tma_load_2d(sB + s * C::B_BYTES, &tmB, &full[s], kb * BK, b0);
          tma_load_2d(sB + s * C::B_BYTES + C::B_BYTES / 2, &tmB, &full[s], kb * BK, b1);
          ++issued;
          if (++s == C::STAGES) { s = 0; ph ^= 1u; }
        }
      }
      if (!ok) {
        // Let the copies already in flight land before the CTA can exit: the
        // last min(issued, STAGES) stages were armed and not re-armed since.
        int n = min(issued, C::STAGES);
        int ss = s;
        uint32_t pp = ph;
        for (int i = 0; i < n; ++i) {
          if (--ss < 0) { ss = C::STAGES - 1; pp ^= 1u; }
          mbar_wait(&full[ss], pp, err);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (one thread)
    if (lane == 0) {
      constexpr uint32_t IDESC = umma_idesc_bf16_f32(BM, BN);
      int s = 0;
      uint32_t ph = 0;
      int it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < total && ok; t += gridDim.x, ++it) {
        const int acc = it & 1;
        const uint32_t aph = (it >> 1) & 1;
        if (!mbar_wait(&tempty[acc], aph ^ 1u, err)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(&full[s], ph, err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + s * C::A_BYTES);
          const uint32_t b0 = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            umma_bf16(d_tmem, umma_desc_sw128(a0 + k * 32), umma_desc_sw128(b0 + k * 32), IDESC,
                      (kb | k) != 0 ? 1u : 0u);
          }
          umma_commit(&empty[s]);
          if (++s == C::STAGES) { s = 0; ph ^= 1u; }
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
      }
      // All MMAs issued by this thread have completed once `done` flips.
      umma_commit(done);
      mbar_wait(done, 0, err);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int quad = warp & 3;  // TMEM lane quadrant this warp may access
    int it = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++it) {
      const int acc = it & 1;
      const uint32_t aph = (it >> 1) & 1;
      if (!mbar_wait_warp(&tfull[acc], aph, err)) break;
      tc_fence_after();
      const int mb = t % num_m, nb = t / num_m;
      const int row = mb * BM + quad * 32 + lane;
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + acc * BN;
      epilogue_tile<BN, EPI>(args.e, taddr, row, row < M, nb, err);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// CTA-pair variant (cta_group::2): a cluster of two CTAs on two SMs computes a
// 256 x BN tile with M = 256 MMAs issued by the even CTA.  Each CTA stages its
// own 128 rows of A and half of the BN rows of B (so each SM fetches half the
// B bytes of the single-CTA tile), and holds the fp32 accumulator of its own
// 128 rows in its TMEM.  Both CTAs' TMA loads complete on the even CTA's
// full barrier; the MMA commits multicast to both CTAs' empty / tmem-full
// barriers; both CTAs' epilogues release the accumulator on the even CTA's
// tmem-empty barrier.
template <int BN>
struct Cfg2 {
  static constexpr uint32_t A_BYTES = BM * BK * 2;
  static constexpr uint32_t B_BYTES = (BN / 2) * BK * 2;
  static constexpr int STAGES = (BN == 256) ? 6 : 8;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
  static constexpr size_t SMEM = 1024 + STAGES * (A_BYTES + B_BYTES) + 256;
};

template <int BN, int EPI>
__global__ void __launch_bounds__(192, 1)
gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const KArgs args) {
  using C = Cfg2<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + C::STAGES * C::B_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tfull = empty + C::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* done = tempty + 2;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(done + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = (rank == 0);
  int* err = args.err;

  int M = args.M_cap;
  if (args.M_dev) M = min(M, __ldg(args.M_dev));
  if (M < 0) M = 0;
  const int num_m = (M + 2 * BM - 1) / (2 * BM);
  const int num_n = args.N_acc / BN;
  const int total = num_m * num_n;
  const int KB = args.K / BK;
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 8);
    }
    mbar_init(done, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(tslot, C::TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem_base = *tslot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer (both CTAs)
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      int s = 0;
      uint32_t ph = 0;
      for (int t = pair; t < total; t += npairs) {
        const int mb = t % num_m, nb = t / num_m;
        const int a_row = mb * 2 * BM + (int)rank * BM;
        int b_row;
        if (EPI == EPI_SWIGLU_BF16)
          b_row = (rank == 0 ? 0 : args.e.up_off) + nb * (BN / 2);
        else
          b_row = nb * BN + (int)rank * (BN / 2);
        bool ok = true;
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(&empty[s], ph ^ 1u, err)) { ok = false; break; }
          if (leader) mbar_arrive_expect_tx(&full[s], 2 * (C::A_BYTES + C::B_BYTES));
          const uint32_t bar = mapa_shared(smem_u32(&full[s]), 0);
          tma_load_2d_pair(sA + s * C::A_BYTES, &tmA, bar, kb * BK, a_row);
          tma_load_2d_pair(sB + s * C::B_BYTES, &tmB, bar, kb * BK, b_row);
          if (++s == C::STAGES) { s = 0; ph ^= 1u; }
        }
        if (!ok) break;
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (one thread of the even CTA)
    if (leader && lane == 0) {
      constexpr uint32_t IDESC = umma_idesc_bf16_f32(2 * BM, BN);
      int s = 0;
      uint32_t ph = 0;
      int it = 0;
      bool ok = true;
      for (int t = pair; t < total && ok; t += npairs, ++it) {
        const int acc = it & 1;
        const uint32_t aph = (it >> 1) & 1;
        if (!mbar_wait_cluster(&tempty[acc], aph ^ 1u, err)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait_cluster(&full[s], ph, err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + s * C::A_BYTES);
          const uint32_t b0 = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            umma_bf16_pair(d_tmem, umma_desc_sw128(a0 + k * 32), umma_desc_sw128(b0 + k * 32), IDESC,
                           (kb | k) != 0 ? 1u : 0u);
          }
          umma_commit_pair(&empty[s], (uint16_t)0x3);
          if (++s == C::STAGES) { s = 0; ph ^= 1u; }
        }
        if (!ok) break;
        umma_commit_pair(&tfull[acc], (uint16_t)0x3);
      }
      umma_commit_pair(done, (uint16_t)0x1);
      mbar_wait(done, 0, err);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue (both CTAs)
    const int quad = warp & 3;
    int it = 0;
    for (int t = pair; t < total; t += npairs, ++it) {
      const int acc = it & 1;
      const uint32_t aph = (it >> 1) & 1;
      if (!mbar_wait_cluster_warp(&tfull[acc], aph, err)) break;
      tc_fence_after();
      const int mb = t % num_m, nb = t / num_m;
      const int row = mb * 2 * BM + (int)rank * BM + quad * 32 + lane;
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + acc * BN;
      epilogue_tile<BN, EPI>(args.e, taddr, row, row < M, nb, err);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(&tempty[acc]), 0));
    }
  }

  tc_fence_before();
  cluster_sync_all();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, C::TMEM_COLS);
  }
}

template <int BN, int EPI>
cudaError_t launch_pair(const CUtensorMap& A, const CUtensorMap& B, const KArgs& a, int grid,
                        cudaStream_t st) {
  using C = Cfg2<BN>;
  static bool attr_done = false;
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc2_kernel<BN, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(192, 1, 1);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gemm_tc2_kernel<BN, EPI>, A, B, a);
}

template <int BN>
cudaError_t dispatch_pair(const CUtensorMap& A, const CUtensorMap& B, const KArgs& a, int grid,
                          cudaStream_t st) {
  switch (a.e.kind) {
    case EPI_BF16: return launch_pair<BN, EPI_BF16>(A, B, a, grid, st);
    case EPI_BF16_ROPE: return launch_pair<BN, EPI_BF16_ROPE>(A, B, a, grid, st);
    case EPI_F32: return launch_pair<BN, EPI_F32>(A, B, a, grid, st);
    case EPI_F32_ACC: return launch_pair<BN, EPI_F32_ACC>(A, B, a, grid, st);
    case EPI_GELU_BF16: return launch_pair<BN, EPI_GELU_BF16>(A, B, a, grid, st);
    case EPI_SWIGLU_BF16: return launch_pair<BN, EPI_SWIGLU_BF16>(A, B, a, grid, st);
    case EPI_SCATTER_BF16: return launch_pair<BN, EPI_SCATTER_BF16>(A, B, a, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

template <int BN, int EPI>
cudaError_t launch_one(const CUtensorMap& A, const CUtensorMap& B, const KArgs& a, int grid,
                       cudaStream_t st) {
  using C = Cfg<BN>;
  static bool attr_done = false;  // per (BN, EPI) instantiation
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  gemm_tc_kernel<BN, EPI><<<grid, 192, C::SMEM, st>>>(A, B, a);
  return cudaGetLastError();
}

template <int BN>
cudaError_t dispatch(const CUtensorMap& A, const CUtensorMap& B, const KArgs& a, int grid,
                     cudaStream_t st) {
  switch (a.e.kind) {
    case EPI_BF16: return launch_one<BN, EPI_BF16>(A, B, a, grid, st);
    case EPI_BF16_ROPE: return launch_one<BN, EPI_BF16_ROPE>(A, B, a, grid, st);
    case EPI_F32: return launch_one<BN, EPI_F32>(A, B, a, grid, st);
    case EPI_F32_ACC: return launch_one<BN, EPI_F32_ACC>(A, B, a, grid, st);
    case EPI_GELU_BF16: return launch_one<BN, EPI_GELU_BF16>(A, B, a, grid, st);
    case EPI_SWIGLU_BF16: return launch_one<BN, EPI_SWIGLU_BF16>(A, B, a, grid, st);
    case EPI_SCATTER_BF16: return launch_one<BN, EPI_SCATTER_BF16>(A, B, a, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

// Tile width of the CTA-pair variant for a GEMM, or 0 for the single-CTA one.
// Pairs with 256-wide tiles wherever M reaches a pair tile: measured on the
// 7B-dims prefill they beat the single-CTA kernel on every GEMM, while 128-wide
// pair tiles lose (the MMA issue per stage no longer hides behind the MMA).
// SP_GEMM_PAIRS=0 in the environment selects the single-CTA kernel (A/B runs);
// SP_GEMM_PAIRS=1 allows 128-wide pair tiles where the column-tile count is small.
int gemm_pair_policy(int M_cap, int N_acc, int kind) {
  static int mode = -1;
  if (mode < 0) {
    const char* s = getenv("SP_GEMM_PAIRS");
    mode = s ? atoi(s) : 2;
  }
  if (mode == 0 || M_cap < 2 * BM) return 0;
  if (N_acc % 256 == 0 && (mode == 2 || N_acc / 256 >= 20 || kind == EPI_SWIGLU_BF16)) return 256;
  return (N_acc % 128 == 0 && mode == 1) ? 128 : 0;
}

bool make_gemm_b(GemmB* b, const void* w, int N, int K, std::string* msg) {
  b->N = N;
  b->K = K;
  return encode_tmap_bf16(&b->map128, w, N, K, 64, msg) &&
         encode_tmap_bf16(&b->map256, w, N, K, 128, msg);
}

cudaError_t gemm_bf16(const CUtensorMap& A, int M_cap, const int* M_dev, const GemmB& B, int N_acc,
                      const GemmEpi& e, int* err, cudaStream_t st) {
  if (M_cap <= 0) return cudaSuccess;
  const int sms = device_sm_count();
  const int mt = (M_cap + BM - 1) / BM;
  // Pick the tile width whose last wave is fullest (RoPE heads and the SwiGLU
  // halves need the 256-wide tile to hold whole heads / 128 output columns).
  bool use256 = (N_acc % 256 == 0);
  if (use256 && e.kind != EPI_SWIGLU_BF16 && e.kind != EPI_BF16_ROPE && N_acc % 128 == 0) {
    const int t256 = mt * (N_acc / 256), t128 = mt * (N_acc / 128);
    const double w256 = (double)t256 / (double)(((t256 + sms - 1) / sms) * sms);
    const double w128 = (double)t128 / (double)(((t128 + sms - 1) / sms) * sms);
    if (w128 > w256 + 0.15) use256 = false;
  }
  if (e.kind == EPI_BF16_ROPE && e.head_dim == 64 && N_acc % 256 != 0) use256 = false;
  KArgs a;
  a.M_cap = M_cap;
  a.M_dev = M_dev;
  a.N_acc = N_acc;
  a.K = B.K;
  a.e = e;
  a.err = err;
  cudaError_t r;
  const int pair_bn = gemm_pair_policy(M_cap, N_acc, e.kind);
  if (pair_bn) {
    const int mp = (M_cap + 2 * BM - 1) / (2 * BM);
    const int tiles = mp * (N_acc / pair_bn);
    const int grid = 2 * std::max(1, std::min(tiles, sms / 2));
    prof_begin_launch(st);
    r = pair_bn == 256 ? dispatch_pair<256>(A, B.map256, a, grid, st) : dispatch_pair<128>(A, B.map128, a, grid, st);
    prof_end_launch(st, SP_K_GEMM, 2.0 * (double)M_cap * (double)N_acc * (double)B.K, 0.0);
    return r;
  }
  const int tiles = mt * (N_acc / (use256 ? 256 : 128));
  const int grid = std::max(1, std::min(tiles, sms));
  prof_begin_launch(st);
  r = use256 ? dispatch<256>(A, B.map256, a, grid, st)
             : dispatch<128>(A, B.map128, a, grid, st);
  double flops = 2.0 * (double)M_cap * (double)N_acc * (double)B.K;
  prof_end_launch(st, SP_K_GEMM, flops, 0.0);
  return r;
}

}  // namespace sp
