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
#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

constexpr int BM = 128;
constexpr int BK = 64;
// K blocks of the first work item's weights a CTA asks L2 for before it waits
// on the previous kernel (weights never depend on it): the fetch of the first
// stages overlaps that kernel's tail.
constexpr int kPrefetchBlocks = 8;

// Epilogue staging: per epilogue warp two boxes of 32 rows x 128 bytes
// (128-byte swizzle) that TMA stores (or reduce-adds) to global memory while
// the warp fills the other one.
constexpr uint32_t BOX_BYTES = 32 * 128;
constexpr uint32_t EPI_STAGE_BYTES = 4 * 2 * BOX_BYTES;

template <int BN>
struct Cfg {
  // BN = 32: the weight-streaming variant (16 KB of weights per stage, deep ring)
  static constexpr int STAGES = (BN == 256) ? 4 : (BN == 32 ? 9 : 6);
  static constexpr uint32_t A_BYTES = BM * BK * 2;
  static constexpr uint32_t B_BYTES = BN * BK * 2;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
  static constexpr size_t SMEM = 1024 + STAGES * (A_BYTES + B_BYTES) + EPI_STAGE_BYTES + 256;
};

struct KArgs {
  int M_cap;
  const int* M_dev;
  int N_acc;       // accumulator columns over the whole GEMM
  int K;
  GemmEpi e;
  int* err;
  int a_seg;       // A k-segment remap (GemmASplit); 0: none
  uint32_t a_map;
  int ksplit;      // single-CTA kernel: K ranges per tile (> 1: fp32 partials to tmO at row s * m_pad)
  int m_pad;       // rows per partial plane (multiple of 32)
  int swiglu_b;    // load B as SwiGLU gate | up halves whatever the epilogue
  float* sk_part;  // pair kernel: stream-K partial tiles [pairs][256][BN] (NULL: whole tiles only)
  int* sk_flags;   // pair kernel: [pairs][8] ready flags, zero between launches
  const int* a_rows;  // A row r is row a_rows[r] of A's map (a row-gather map); NULL: r
};

// Column of A's tensor map holding the GEMM's k-coordinate k.
SP_DEVINL int a_col(const KArgs& a, int k) {
  if (a.a_seg == 0) return k;
  const int s = k / a.a_seg;
  return (int)((a.a_map >> (4 * s)) & 15u) * a.a_seg + (k - s * a.a_seg);
}

// Partial sums other pairs computed for this tile (stream-K tail): `n` slots,
// `stride` floats apart, from the slot of the first.  A slot holds a 256-row
// tile as float4 [BN/32 column chunks][8][256 rows], so that a warp's 32 rows
// of one float4 column are 512 contiguous bytes.
struct Fix {
  const float* p = nullptr;
  int n = 0;
  size_t stride = 0;
  int rit = 0;  // this lane's row within the 256-row tile
};

SP_DEVINL void fix_add(const Fix& f, int col, float (&v)[32]) {
#pragma unroll 1
  for (int q = 0; q < f.n; ++q) {
    const float4* s = reinterpret_cast<const float4*>(f.p + q * f.stride) + (size_t)(col >> 5) * 8 * 256 + f.rit;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 x = __ldcg(s + j * 256);
      v[4 * j] += x.x;
      v[4 * j + 1] += x.y;
      v[4 * j + 2] += x.z;
      v[4 * j + 3] += x.w;
    }
  }
}

// Completes a tcgen05.ld of 32 columns into v and adds the partials of those
// columns; the first partial's loads are issued before the TMEM wait so the
// two latencies overlap.
SP_DEVINL void fix_add_waited(const Fix& f, int col, float (&v)[32]) {
  if (f.n == 0) {
    tmem_ld_wait();
    return;
  }
  float4 x[8];
  const float4* s = reinterpret_cast<const float4*>(f.p) + (size_t)(col >> 5) * 8 * 256 + f.rit;
#pragma unroll
  for (int j = 0; j < 8; ++j) x[j] = __ldcg(s + j * 256);
  tmem_ld_wait();
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    v[4 * j] += x[j].x;
    v[4 * j + 1] += x[j].y;
    v[4 * j + 2] += x[j].z;
    v[4 * j + 3] += x[j].w;
  }
  if (f.n > 1) {
    Fix rest = f;
    rest.p = f.p + f.stride;
    rest.n = f.n - 1;
    fix_add(rest, col, v);
  }
}

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
SP_DEVINL void epilogue_tile(const GemmEpi& e, uint32_t taddr, int row, bool live, int nb, int* err,
                             const Fix& fx) {
  float v[32];

  if (EPI == EPI_SWIGLU_BF16) {
    float u[32];
#pragma unroll 1
    for (int c = 0; c < BN / 64; ++c) {
      tmem_ld_32x32b_x32(taddr + c * 32, v);
      tmem_ld_32x32b_x32(taddr + BN / 2 + c * 32, u);
      tmem_ld_wait();
      if (live) {
        fix_add(fx, c * 32, v);
        fix_add(fx, BN / 2 + c * 32, u);
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
            fix_add(fx, hb + c, v);
            fix_add(fx, hb + half + c, u);
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
            fix_add(fx, hb + c, v);
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
      fix_add(fx, c * 32, v);
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

// One 16-byte chunk of this lane's row of a staging box (128-byte swizzle:
// chunk q of row r sits at chunk q ^ (r % 8), so the 8 rows a shared-memory
// wavefront serves hit 8 different bank groups).
SP_DEVINL void box_put(uint8_t* box, int lane, int q, uint4 w) {
  *reinterpret_cast<uint4*>(box + lane * 128 + ((q ^ (lane & 7)) << 4)) = w;
}

// 32 fp32 values as bf16 into half h (64 bytes) of this lane's box row.
SP_DEVINL void box_put_bf16_half(uint8_t* box, int lane, int h, const float (&v)[32]) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint4 u;
    u.x = pack_bf16x2(v[8 * q + 0], v[8 * q + 1]);
    u.y = pack_bf16x2(v[8 * q + 2], v[8 * q + 3]);
    u.z = pack_bf16x2(v[8 * q + 4], v[8 * q + 5]);
    u.w = pack_bf16x2(v[8 * q + 6], v[8 * q + 7]);
    box_put(box, lane, 4 * h + q, u);
  }
}

SP_DEVINL void zero32(float (&v)[32]) {
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = 0.f;
}

// Hands the filled box(es) of this warp to TMA: every lane's shared-memory
// writes are made visible to the async proxy, then lane 0 issues the copies
// as one bulk group.
SP_DEVINL void box_fence(int lane) {
  fence_proxy_async_smem();
  __syncwarp();
}

// Drains this warp's 32 rows (row0 + lane) of a BN-wide accumulator tile
// from TMEM, applies the epilogue and writes it with TMA through the staging
// boxes `boxes` (two per warp; `nbox` counts the boxes issued so far).  Rows
// past M are written as zeros (EPI_F32_ACC: adds zero); rows past the output
// map's extent are clipped by TMA.
template <int BN, int EPI>
SP_DEVINL void epilogue_tma(const GemmEpi& e, const CUtensorMap* tmO, uint32_t taddr, int row0, int lane,
                            bool live, int nb, uint8_t* boxes, int& nbox, const Fix& fx, int* err) {
  float v[32];
  if (EPI == EPI_F32 || EPI == EPI_F32_ACC) {
#pragma unroll 1
    for (int c = 0; c < BN / 32; ++c) {
      tmem_ld_32x32b_x32(taddr + c * 32, v);
      fix_add_waited(fx, c * 32, v);
      if (!live) zero32(v);
      if (lane == 0) bulk_wait_read<1>();
      __syncwarp();
      uint8_t* box = boxes + (nbox & 1) * BOX_BYTES;
#pragma unroll
      for (int q = 0; q < 8; ++q)
        box_put(box, lane, q, make_uint4(__float_as_uint(v[4 * q]), __float_as_uint(v[4 * q + 1]),
                                         __float_as_uint(v[4 * q + 2]), __float_as_uint(v[4 * q + 3])));
      box_fence(lane);
      if (lane == 0) {
        if (EPI == EPI_F32_ACC)
          tma_reduce_add_2d(tmO, box, nb * BN + c * 32, row0);
        else
          tma_store_2d(tmO, box, nb * BN + c * 32, row0);
        bulk_commit();
      }
      ++nbox;
    }
  } else if (EPI == EPI_BF16 || EPI == EPI_GELU_BF16) {
#pragma unroll 1
    for (int c2 = 0; c2 < BN / 64; ++c2) {
      if (lane == 0) bulk_wait_read<1>();
      __syncwarp();
      uint8_t* box = boxes + (nbox & 1) * BOX_BYTES;
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        tmem_ld_32x32b_x32(taddr + c2 * 64 + h * 32, v);
        fix_add_waited(fx, c2 * 64 + h * 32, v);
        if (EPI == EPI_GELU_BF16) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = gelu_erf(v[i]);
        }
        if (!live) zero32(v);
        box_put_bf16_half(box, lane, h, v);
      }
      box_fence(lane);
      if (lane == 0) {
        tma_store_2d(tmO, box, nb * BN + c2 * 64, row0);
        bulk_commit();
      }
      ++nbox;
    }
  } else if (EPI == EPI_SWIGLU_BF16) {
    // accumulator columns [0, BN/2) gate, [BN/2, BN) up -> BN/2 output columns
    float u[32];
#pragma unroll 1
    for (int c2 = 0; c2 < BN / 128; ++c2) {
      if (lane == 0) bulk_wait_read<1>();
      __syncwarp();
      uint8_t* box = boxes + (nbox & 1) * BOX_BYTES;
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        const int c = c2 * 64 + h * 32;
        tmem_ld_32x32b_x32(taddr + c, v);
        tmem_ld_32x32b_x32(taddr + BN / 2 + c, u);
        fix_add_waited(fx, c, v);
        fix_add(fx, BN / 2 + c, u);
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = silu(v[i]) * u[i];
        if (!live) zero32(v);
        box_put_bf16_half(box, lane, h, v);
      }
      box_fence(lane);
      if (lane == 0) {
        tma_store_2d(tmO, box, nb * (BN / 2) + c2 * 64, row0);
        bulk_commit();
      }
      ++nbox;
    }
  } else if (EPI == EPI_BF16_ROPE) {
    // per head of dh = 64 or 128 columns: dh / 64 boxes; rotate-half pairs
    // column c of the first half with column c + dh/2
    const int dh = e.head_dim;
    const int half = dh >> 1;
    const int row = row0 + lane;
    const int p = live ? __ldg(e.pos + row) : 0;
    const bool pos_ok = p >= 0 && p < e.max_pos;
    if (live && !pos_ok) set_error(err, SP_DEVERR_INDEX);
    const int nbx = dh >> 6;
    float u[32];
#pragma unroll 1
    for (int hb = 0; hb < BN; hb += dh) {
      const int col0 = nb * BN + hb;
      if (lane == 0) {
        if (nbx == 2) bulk_wait_read<0>(); else bulk_wait_read<1>();
      }
      __syncwarp();
      uint8_t* bx0 = boxes + (nbox & 1) * BOX_BYTES;
      uint8_t* bx1 = boxes + ((nbox + 1) & 1) * BOX_BYTES;
      if (col0 < e.rope_cols) {
#pragma unroll 1
        for (int c = 0; c < half; c += 32) {
          tmem_ld_32x32b_x32(taddr + hb + c, v);
          tmem_ld_32x32b_x32(taddr + hb + half + c, u);
          fix_add_waited(fx, hb + c, v);
          fix_add(fx, hb + half + c, u);
          if (live) {
            const float4* cs = reinterpret_cast<const float4*>(e.rope + (size_t)(pos_ok ? p : 0) * half + c);
#pragma unroll
            for (int i2 = 0; i2 < 16; ++i2) {
              const float4 r = __ldg(cs + i2);
              const float a0 = v[2 * i2], b0 = u[2 * i2], a1 = v[2 * i2 + 1], b1 = u[2 * i2 + 1];
              v[2 * i2] = a0 * r.x - b0 * r.y;
              u[2 * i2] = b0 * r.x + a0 * r.y;
              v[2 * i2 + 1] = a1 * r.z - b1 * r.w;
              u[2 * i2 + 1] = b1 * r.z + a1 * r.w;
            }
          } else {
            zero32(v);
            zero32(u);
          }
          const int ov = c, ou = c + half;  // output offsets within the head
          box_put_bf16_half((ov >> 6) ? bx1 : bx0, lane, (ov >> 5) & 1, v);
          box_put_bf16_half((ou >> 6) ? bx1 : bx0, lane, (ou >> 5) & 1, u);
        }
      } else {
#pragma unroll 1
        for (int o = 0; o < dh; o += 32) {
          tmem_ld_32x32b_x32(taddr + hb + o, v);
          fix_add_waited(fx, hb + o, v);
          if (!live) zero32(v);
          box_put_bf16_half((o >> 6) ? bx1 : bx0, lane, (o >> 5) & 1, v);
        }
      }
      box_fence(lane);
      if (lane == 0) {
        tma_store_2d(tmO, bx0, col0, row0);
        if (nbx == 2) tma_store_2d(tmO, bx1, col0 + 64, row0);
        bulk_commit();
      }
      nbox += nbx;
    }
  }
}

template <int BN, int EPI>
__global__ void __launch_bounds__(192, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmO,
               const KArgs args) {
  using C = Cfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint8_t* sE = sB + C::STAGES * C::B_BYTES;  // epilogue staging boxes (1024-byte aligned)
  uint64_t* full = reinterpret_cast<uint64_t*>(sE + EPI_STAGE_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tfull = empty + C::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* done = tempty + 2;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(done + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  int* err = args.err;

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
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    // the weight boxes of this CTA's first work item (tile order from the host
    // cap M_cap; a wrong guess only wastes the hint).  BN = 32 is the
    // weight-streaming variant, whose weights are A.
    const int nm0 = (args.M_cap + BM - 1) / BM;
    const int ks0 = args.ksplit > 1 ? args.ksplit : 1;
    const int t0 = blockIdx.x;
    if (t0 < nm0 * (args.N_acc / BN) * ks0) {
      const int tile = t0 / ks0, sp = t0 - tile * ks0;
      const int mb = tile % nm0, nb = tile / nm0;
      const int KB0 = args.K / BK;
      const int kb0 = sp * KB0 / ks0, kb1 = min((sp + 1) * KB0 / ks0, kb0 + kPrefetchBlocks);
      const bool sw = (EPI == EPI_SWIGLU_BF16) || args.swiglu_b;
      for (int kb = kb0; kb < kb1; ++kb) {
        if (BN == 32) {
          tma_prefetch_l2_2d(&tmA, kb * BK, mb * BM);
        } else {
          tma_prefetch_l2_2d(&tmB, kb * BK, sw ? nb * (BN / 2) : nb * BN);
          tma_prefetch_l2_2d(&tmB, kb * BK, sw ? args.e.up_off + nb * (BN / 2) : nb * BN + BN / 2);
        }
      }
    }
  }
  // everything above overlaps the previous kernel's tail (programmatic launch)
  pdl_wait();
  pdl_trigger();

  int M = args.M_cap;
  if (args.M_dev) M = min(M, __ldg(args.M_dev));
  if (M < 0) M = 0;
  const int num_m = (M + BM - 1) / BM;
  const int num_n = args.N_acc / BN;
  const int ks = args.ksplit > 1 ? args.ksplit : 1;
  const int total = num_m * num_n * ks;  // work items: (tile, K range)
  const int KB = args.K / BK;
  const bool swb = (EPI == EPI_SWIGLU_BF16) || args.swiglu_b;

  if (warp == 0 && args.a_rows) {
    // ------------------------------------------------------------ producer, A rows gathered
    // Each lane copies four of the tile's 128 A rows per K block with one
    // tile::gather4 load (its map's box is 64 columns by one row); lane 0 arms
    // the stage and loads B.  Rows past M read row 0 (their results are not
    // stored); a row index outside A's map reads zeros.
    int s = 0;
    uint32_t ph = 0;
    int issued = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
      const int tile = t / ks, sp = t - tile * ks;
      const int mb = tile % num_m, nb = tile / num_m;
      const int m0 = mb * BM;
      int b0, b1;
      if (swb) {
        b0 = nb * (BN / 2);
        b1 = args.e.up_off + nb * (BN / 2);
      } else {
        b0 = nb * BN;
        b1 = nb * BN + BN / 2;
      }
      int r[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int row = m0 + 4 * lane + q;
        r[q] = row < M ? __ldg(args.a_rows + row) : 0;
      }
      const int kb0 = sp * KB / ks, kb1 = (sp + 1) * KB / ks;
      for (int kb = kb0; kb < kb1; ++kb) {
        if (!mbar_wait_warp(&empty[s], ph ^ 1u, err)) { ok = false; break; }
        if (lane == 0) {
          mbar_arrive_expect_tx(&full[s], C::A_BYTES + C::B_BYTES);
          tma_load_2d(sB + s * C::B_BYTES, &tmB, &full[s], kb * BK, b0);
          tma_load_2d(sB + s * C::B_BYTES + C::B_BYTES / 2, &tmB, &full[s], kb * BK, b1);
        }
        __syncwarp();
        tma_gather4_2d(sA + s * C::A_BYTES + lane * (4 * BK * 2), &tmA, &full[s], a_col(args, kb * BK), r[0], r[1],
                       r[2], r[3]);
        ++issued;
        if (++s == C::STAGES) { s = 0; ph ^= 1u; }
      }
    }
    if (!ok && lane == 0) {
      // the copies already in flight land before the CTA can exit
      int n = min(issued, C::STAGES);
      int ss = s;
      uint32_t pp = ph;
      for (int i = 0; i < n; ++i) {
        if (--ss < 0) { ss = C::STAGES - 1; pp ^= 1u; }
        mbar_wait(&full[ss], pp, err);
      }
    }
  } else if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0;
      int issued = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
        const int tile = t / ks, sp = t - tile * ks;
        const int mb = tile % num_m, nb = tile / num_m;
        const int m0 = mb * BM;
        int b0, b1;
        if (swb) {
          b0 = nb * (BN / 2);
          b1 = args.e.up_off + nb * (BN / 2);
        } else {
          b0 = nb * BN;
          b1 = nb * BN + BN / 2;
        }
        const int kb0 = sp * KB / ks, kb1 = (sp + 1) * KB / ks;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&empty[s], ph ^ 1u, err)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[s], C::A_BYTES + C::B_BYTES);
          tma_load_2d(sA + s * C::A_BYTES, &tmA, &full[s], a_col(args, kb * BK), m0);
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
        const int sp = t % ks;
        const int kb0 = sp * KB / ks, kb1 = (sp + 1) * KB / ks;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&full[s], ph, err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + s * C::A_BYTES);
          const uint32_t b0 = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            umma_bf16(d_tmem, umma_desc_sw128(a0 + k * 32), umma_desc_sw128(b0 + k * 32), IDESC,
                      (kb != kb0 || k != 0) ? 1u : 0u);
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
    uint8_t* boxes = sE + quad * 2 * BOX_BYTES;
    int nbox = 0;
    int it = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++it) {
      const int acc = it & 1;
      const uint32_t aph = (it >> 1) & 1;
      if (!mbar_wait_warp(&tfull[acc], aph, err)) break;
      tc_fence_after();
      const int tile = t / ks, sp = t - tile * ks;
      const int mb = tile % num_m, nb = tile / num_m;
      const int row0 = mb * BM + quad * 32;
      const int row = row0 + lane;
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + acc * BN;
      if (ks > 1) {
        // a K range: its raw fp32 partial into plane sp (rows past m_pad belong to the next plane)
        if (EPI == EPI_F32 && row0 < args.m_pad)
          epilogue_tma<BN, EPI>(args.e, &tmO, taddr, sp * args.m_pad + row0, lane, row < M, nb, boxes, nbox, Fix(),
                                err);
      } else if (EPI == EPI_SCATTER_BF16) {
        epilogue_tile<BN, EPI>(args.e, taddr, row, row < M, nb, err, Fix());
      } else {
        epilogue_tma<BN, EPI>(args.e, &tmO, taddr, row0, lane, row < M, nb, boxes, nbox, Fix(), err);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
    }
    if (lane == 0) bulk_wait<0>();  // the staging boxes stay valid until every copy is done
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}


// Work split of the pair kernel over its W pairs.  Whole tiles go round-robin
// while every pair gets one (data-parallel waves); when the last, partial
// wave would leave at least half of the pairs idle, its r tiles are instead
// cut along K into s = min(W / r, kSkMaxSplit) equal ranges spread over r*s
// pairs (a stream-K tail, after Osama et al., PPoPP 2023).  The pair with a
// tile's first K range finishes the tile after adding the fp32 partials the
// other s - 1 pairs wrote to their slots.  The general form below also
// allows ranges that straddle tiles (at most two fragments per pair: the end
// of one tile, written as a partial, and the start of the next).
constexpr int kSkMinIters = 8;   // K blocks per tail range at least (fix-up traffic vs balance)
constexpr int kSkMaxSplit = 2;   // one partial per tile: the finishing epilogue waits on one pair

struct Sched {
  int num_m, KB, W, p;
  int full;        // tiles of the data-parallel waves
  int Wt;          // pairs sharing the tail (0: no tail)
  long long I;     // K-block iterations of the tail
  SP_DEVINL long long bnd(int q) const { return (long long)q * I / Wt; }
};

struct Frag {
  int t, k0, k1;
  int kind;        // 0 whole tile, 1 first K range (finishes the tile), 2 later K range (partial)
};

SP_DEVINL Sched make_sched(int total, int num_m, int KB, int W, int p, bool stream_k) {
  Sched s;
  s.num_m = num_m;
  s.KB = KB;
  s.W = W;
  s.p = p;
  s.full = total;
  s.Wt = 0;
  s.I = 0;
  const int r = total % W;
  if (stream_k && r != 0) {
    const long long I = (long long)r * KB;
    const int split = min(min(W / r, kSkMaxSplit), KB / kSkMinIters);
    const int Wt = r * split;
    if (split > 1) {
      s.full = total - r;
      s.Wt = Wt;
      s.I = I;
    }
  }
  return s;
}

struct Cursor {
  int j = 0;
  long long g = -1;
};

SP_DEVINL bool sched_next(const Sched& s, Cursor& c, Frag& f) {
  const int t = s.p + c.j * s.W;
  if (t < s.full) {
    f.t = t;
    f.k0 = 0;
    f.k1 = s.KB;
    f.kind = 0;
    ++c.j;
    return true;
  }
  if (s.p >= s.Wt) return false;
  if (c.g < 0) c.g = s.bnd(s.p);
  const long long e = s.bnd(s.p + 1);
  if (c.g >= e) return false;
  const int tl = (int)(c.g / s.KB);
  const int k0 = (int)(c.g - (long long)tl * s.KB);
  const int k1 = (int)min((long long)s.KB, (long long)k0 + (e - c.g));
  f.t = s.full + tl;
  f.k0 = k0;
  f.k1 = k1;
  f.kind = k0 > 0 ? 2 : (k1 < s.KB ? 1 : 0);
  c.g += k1 - k0;
  return true;
}

// Pairs after `p` whose first tail fragment belongs to tail tile `t`.
SP_DEVINL int sched_contributors(const Sched& s, int t) {
  const long long g1 = (long long)(t - s.full + 1) * s.KB;
  int n = 0;
  for (int q = s.p + 1; q < s.Wt && s.bnd(q) < g1; ++q) ++n;
  return n;
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
  static constexpr size_t SMEM = 1024 + STAGES * (A_BYTES + B_BYTES) + EPI_STAGE_BYTES + 256;
};

template <int BN, int EPI>
__global__ void __launch_bounds__(192, 1)
gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmO,
                const KArgs args) {
  using C = Cfg2<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint8_t* sE = sB + C::STAGES * C::B_BYTES;  // epilogue staging boxes (1024-byte aligned)
  uint64_t* full = reinterpret_cast<uint64_t*>(sE + EPI_STAGE_BYTES);
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
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    // this CTA's half of the B (weight) rows of the pair's first tile (tile
    // order from the host cap M_cap; a wrong guess only wastes the hint)
    const int nm0 = (args.M_cap + 2 * BM - 1) / (2 * BM);
    const int pair0 = blockIdx.x >> 1;
    if (pair0 < nm0 * (args.N_acc / BN)) {
      const int nb = pair0 / nm0;
      const int b_row = (EPI == EPI_SWIGLU_BF16) ? (rank == 0 ? 0 : args.e.up_off) + nb * (BN / 2)
                                                 : nb * BN + (int)rank * (BN / 2);
      const int kb1 = min(args.K / BK, kPrefetchBlocks);
      for (int kb = 0; kb < kb1; ++kb) tma_prefetch_l2_2d(&tmB, kb * BK, b_row);
    }
  }
  // everything above overlaps the previous kernel's tail (programmatic launch)
  pdl_wait();
  pdl_trigger();

  int M = args.M_cap;
  if (args.M_dev) M = min(M, __ldg(args.M_dev));
  if (M < 0) M = 0;
  const int num_m = (M + 2 * BM - 1) / (2 * BM);
  const int num_n = args.N_acc / BN;
  const int total = num_m * num_n;
  const int KB = args.K / BK;
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  const Sched sc = make_sched(total, num_m, KB, npairs, pair, args.sk_part != nullptr && args.sk_flags != nullptr);

  if (warp == 0 && args.a_rows) {
    // ------------------------------------------------------------ producer (both CTAs), A rows gathered
    // As the single-CTA kernel's: each lane copies four of this CTA's 128 A
    // rows per K block (tile::gather4, the pair form signalling the even CTA's
    // barrier); lane 0 waits, arms (even CTA) and loads this CTA's B half.
    int s = 0;
    uint32_t ph = 0;
    Cursor cur;
    Frag f;
    while (sched_next(sc, cur, f)) {
      const int mb = f.t % num_m, nb = f.t / num_m;
      const int a_row = mb * 2 * BM + (int)rank * BM;
      int b_row;
      if (EPI == EPI_SWIGLU_BF16)
        b_row = (rank == 0 ? 0 : args.e.up_off) + nb * (BN / 2);
      else
        b_row = nb * BN + (int)rank * (BN / 2);
      int r[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int row = a_row + 4 * lane + q;
        r[q] = row < M ? __ldg(args.a_rows + row) : 0;
      }
      bool ok = true;
      for (int kb = f.k0; kb < f.k1; ++kb) {
        if (!mbar_wait_warp(&empty[s], ph ^ 1u, err)) { ok = false; break; }
        const uint32_t bar = mapa_shared(smem_u32(&full[s]), 0);
        if (lane == 0) {
          if (leader) mbar_arrive_expect_tx(&full[s], 2 * (C::A_BYTES + C::B_BYTES));
          tma_load_2d_pair(sB + s * C::B_BYTES, &tmB, bar, kb * BK, b_row);
        }
        __syncwarp();
        tma_gather4_2d_pair(sA + s * C::A_BYTES + lane * (4 * BK * 2), &tmA, bar, a_col(args, kb * BK), r[0], r[1],
                            r[2], r[3]);
        if (++s == C::STAGES) { s = 0; ph ^= 1u; }
      }
      if (!ok) break;
    }
  } else if (warp == 0) {
    // ------------------------------------------------------------ producer (both CTAs)
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0;
      Cursor cur;
      Frag f;
      while (sched_next(sc, cur, f)) {
        const int mb = f.t % num_m, nb = f.t / num_m;
        const int a_row = mb * 2 * BM + (int)rank * BM;
        int b_row;
        if (EPI == EPI_SWIGLU_BF16)
          b_row = (rank == 0 ? 0 : args.e.up_off) + nb * (BN / 2);
        else
          b_row = nb * BN + (int)rank * (BN / 2);
        bool ok = true;
        for (int kb = f.k0; kb < f.k1; ++kb) {
          if (!mbar_wait(&empty[s], ph ^ 1u, err)) { ok = false; break; }
          if (leader) mbar_arrive_expect_tx(&full[s], 2 * (C::A_BYTES + C::B_BYTES));
          const uint32_t bar = mapa_shared(smem_u32(&full[s]), 0);
          tma_load_2d_pair(sA + s * C::A_BYTES, &tmA, bar, a_col(args, kb * BK), a_row);
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
      Cursor cur;
      Frag f;
      for (; ok && sched_next(sc, cur, f); ++it) {
        const int acc = it & 1;
        const uint32_t aph = (it >> 1) & 1;
        if (!mbar_wait_cluster(&tempty[acc], aph ^ 1u, err)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = f.k0; kb < f.k1; ++kb) {
          if (!mbar_wait_cluster(&full[s], ph, err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + s * C::A_BYTES);
          const uint32_t b0 = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            umma_bf16_pair(d_tmem, umma_desc_sw128(a0 + k * 32), umma_desc_sw128(b0 + k * 32), IDESC,
                           (kb != f.k0 || k != 0) ? 1u : 0u);
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
    const int rit = (int)rank * BM + quad * 32 + lane;  // row within the 256-row pair tile
    const int fslot = (int)rank * 4 + quad;              // this warp's ready flag within a pair's 8
    const size_t slot_floats = (size_t)2 * BM * BN;
    uint8_t* boxes = sE + quad * 2 * BOX_BYTES;
    int nbox = 0;
    int it = 0;
    Cursor cur;
    Frag f;
    for (; sched_next(sc, cur, f); ++it) {
      const int acc = it & 1;
      const uint32_t aph = (it >> 1) & 1;
      if (!mbar_wait_cluster_warp(&tfull[acc], aph, err)) break;
      tc_fence_after();
      const int mb = f.t % num_m, nb = f.t / num_m;
      const int row0 = mb * 2 * BM + (int)rank * BM + quad * 32;
      const int row = row0 + lane;
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + acc * BN;
      if (f.kind == 2) {
        // a later K range: hand the raw fp32 partial to the pair finishing the tile
        float v[32];
        float4* dst = reinterpret_cast<float4*>(args.sk_part + pair * slot_floats) + rit;
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          tmem_ld_32x32b_x32(taddr + c * 32, v);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 8; ++q)
            __stcg(dst + (size_t)(c * 8 + q) * 256, make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]));
        }
        __threadfence();
        __syncwarp();
        if (lane == 0) st_release_gpu(args.sk_flags + pair * 8 + fslot, 1);
      } else {
        Fix fx;
        if (f.kind == 1) {
          // the first K range: wait for the partials of the pairs that did the rest
          fx.n = sched_contributors(sc, f.t);
          fx.p = args.sk_part + (pair + 1) * slot_floats;
          fx.stride = slot_floats;
          fx.rit = rit;
          for (int q = 0; q < fx.n; ++q) {
            int* flag = args.sk_flags + (pair + 1 + q) * 8 + fslot;
            int ok = 1;
            if (lane == 0) ok = wait_flag(flag, err) ? 1 : 0;
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) { fx.n = q; break; }  // warp-uniform
            (void)ld_acquire_gpu(flag);     // every lane synchronises with the writer's release
            __syncwarp();
            if (lane == 0) *flag = 0;       // the only reader: leave the flags zero for the next launch
          }
        }
        if (EPI == EPI_SCATTER_BF16)
          epilogue_tile<BN, EPI>(args.e, taddr, row, row < M, nb, err, fx);
        else
          epilogue_tma<BN, EPI>(args.e, &tmO, taddr, row0, lane, row < M, nb, boxes, nbox, fx, err);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(&tempty[acc]), 0));
    }
    if (lane == 0) bulk_wait<0>();  // the staging boxes stay valid until every copy is done
  }

  tc_fence_before();
  cluster_sync_all();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, C::TMEM_COLS);
  }
}

constexpr size_t kSlotFloats = (size_t)2 * BM * 256;  // one 256 x 256 fp32 partial tile

// Clusters of the pair kernel that fit on the device at once (0 if unknown).
// The stream-K tail needs every pair resident: a pair finishing a tile waits
// for pairs with higher indices.
template <int BN, int EPI>
int pair_max_clusters() {
  static int cached_dev = -1, n = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev != cached_dev) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2, 1, 1);
    cfg.blockDim = dim3(192, 1, 1);
    cfg.dynamicSmemBytes = Cfg2<BN>::SMEM;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int c = 0;
    if (cudaOccupancyMaxActiveClusters(&c, gemm_tc2_kernel<BN, EPI>, &cfg) != cudaSuccess) {
      (void)cudaGetLastError();
      c = 0;
    }
    n = c;
    cached_dev = dev;
  }
  return n;
}

// tiles: pair tiles for M_cap rows (an upper bound of the device row count).
template <int BN, int EPI>
cudaError_t launch_pair(const CUtensorMap& A, const CUtensorMap& B, const CUtensorMap& O, KArgs a, int tiles,
                        int slots, cudaStream_t st) {
  using C = Cfg2<BN>;
  static bool attr_done = false;
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc2_kernel<BN, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  const int maxc = pair_max_clusters<BN, EPI>();
  const int pairs = std::max(1, std::min(tiles, maxc > 0 ? maxc : device_sm_count() / 2));
  if (maxc <= 0 || pairs > slots) {
    a.sk_part = nullptr;
    a.sk_flags = nullptr;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * pairs, 1, 1);
  cfg.blockDim = dim3(192, 1, 1);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, gemm_tc2_kernel<BN, EPI>, A, B, O, a);
}

template <int BN>
cudaError_t dispatch_pair(const CUtensorMap& A, const CUtensorMap& B, const CUtensorMap& O, const KArgs& a,
                          int tiles, int slots, cudaStream_t st) {
  switch (a.e.kind) {
    case EPI_BF16: return launch_pair<BN, EPI_BF16>(A, B, O, a, tiles, slots, st);
    case EPI_BF16_ROPE: return launch_pair<BN, EPI_BF16_ROPE>(A, B, O, a, tiles, slots, st);
    case EPI_F32: return launch_pair<BN, EPI_F32>(A, B, O, a, tiles, slots, st);
    case EPI_F32_ACC: return launch_pair<BN, EPI_F32_ACC>(A, B, O, a, tiles, slots, st);
    case EPI_GELU_BF16: return launch_pair<BN, EPI_GELU_BF16>(A, B, O, a, tiles, slots, st);
    case EPI_SWIGLU_BF16: return launch_pair<BN, EPI_SWIGLU_BF16>(A, B, O, a, tiles, slots, st);
    case EPI_SCATTER_BF16: return launch_pair<BN, EPI_SCATTER_BF16>(A, B, O, a, tiles, slots, st);
    default: return cudaErrorInvalidValue;
  }
}

// Sum of the K-range partials of a split GEMM (planes of m_pad x N_acc fp32)
// and the epilogue the unsplit GEMM would have fused (one block row per row).
__global__ void __launch_bounds__(256) splitk_reduce_kernel(const float* __restrict__ part, int ks, int m_pad,
                                                            int M_cap, const int* __restrict__ M_dev, int N_acc,
                                                            int BN, const GemmEpi e, int* err) {
  pdl_wait();
  pdl_trigger();
  int M = M_cap;
  if (M_dev) M = min(M, __ldg(M_dev));
  const int row = blockIdx.y;
  if (row >= M) return;
  const size_t plane = (size_t)m_pad * N_acc;
  const float* pr = part + (size_t)row * N_acc;
  auto sum = [&](int c) {
    float v = 0.f;
    for (int s = 0; s < ks; ++s) v += __ldcg(pr + s * plane + c);
    return v;
  };
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (e.kind == EPI_SWIGLU_BF16) {
    if (c >= N_acc / 2) return;
    const int nb = c / (BN / 2), j = c - nb * (BN / 2);
    const float g = sum(nb * BN + j), u = sum(nb * BN + BN / 2 + j);
    reinterpret_cast<__nv_bfloat16*>(e.out)[(size_t)row * e.ldo + c] = __float2bfloat16_rn(silu(g) * u);
    return;
  }
  if (c >= N_acc) return;
  if (e.kind == EPI_BF16_ROPE) {
    const int dh = e.head_dim, half = dh >> 1;
    const int hb = (c / dh) * dh, i = c - hb;
    __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(e.out) + (size_t)row * e.ldo;
    if (hb < e.rope_cols) {
      if (i >= half) return;  // the pair's first element writes both
      const int p = __ldg(e.pos + row);
      const bool pos_ok = p >= 0 && p < e.max_pos;
      if (!pos_ok) set_error(err, SP_DEVERR_INDEX);
      const float2 r = __ldg(e.rope + (size_t)(pos_ok ? p : 0) * half + i);
      const float a = sum(c), b = sum(c + half);
      o[c] = __float2bfloat16_rn(a * r.x - b * r.y);
      o[c + half] = __float2bfloat16_rn(b * r.x + a * r.y);
    } else {
      o[c] = __float2bfloat16_rn(sum(c));
    }
    return;
  }
  const float v = sum(c);
  if (e.kind == EPI_F32) {
    reinterpret_cast<float*>(e.out)[(size_t)row * e.ldo + c] = v;
  } else if (e.kind == EPI_F32_ACC) {
    reinterpret_cast<float*>(e.out)[(size_t)row * e.ldo + c] += v;
  } else if (e.kind == EPI_GELU_BF16) {
    reinterpret_cast<__nv_bfloat16*>(e.out)[(size_t)row * e.ldo + c] = __float2bfloat16_rn(gelu_erf(v));
  } else if (e.kind == EPI_SCATTER_BF16) {
    const int orow = __ldg(e.row_map + row);
    if (orow < 0) {
      set_error(err, SP_DEVERR_INDEX);
      return;
    }
    reinterpret_cast<__nv_bfloat16*>(e.out)[(size_t)orow * e.ldo + c] = __float2bfloat16_rn(v);
  } else {
    reinterpret_cast<__nv_bfloat16*>(e.out)[(size_t)row * e.ldo + c] = __float2bfloat16_rn(v);
  }
}

// Sum of the K-range partials of the weight-streaming GEMM and the epilogue
// of the unsplit GEMM.  Partials are planes [ks][N_acc][32]: row n = output
// column n (weight row), column m = activation row m.  Thread (c, q): output
// column c, activation rows 8q..8q+7 (a warp reads 8 consecutive 128-byte
// partial rows; its stores cover 8 consecutive columns of 4 rows).
__global__ void __launch_bounds__(256) splitk_reduce_t_kernel(const float* __restrict__ part, int ks, int N_acc,
                                                              int M_cap, const int* __restrict__ M_dev,
                                                              int cols, const GemmEpi e, int* err) {
  pdl_wait();
  pdl_trigger();
  int M = M_cap;
  if (M_dev) M = min(M, __ldg(M_dev));
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  const int c = t >> 2, m0 = (t & 3) * 8;
  if (c >= cols || m0 >= M) return;
  const int mn = min(8, M - m0);
  const size_t plane = (size_t)N_acc * 32;
  // Sums 8 rows of NC columns over the ks ranges, in range order.  The loads
  // of four ranges (for every column) go out before their adds, so a thread
  // waits on L2 about ks / 4 times instead of ks * NC times.
  auto sum_cols = [&](auto nc_tag, const int* n, float (*v)[8]) {
    constexpr int NC = decltype(nc_tag)::value;
    const float* p[NC];
#pragma unroll
    for (int k = 0; k < NC; ++k) {
      p[k] = part + (size_t)n[k] * 32 + m0;
#pragma unroll
      for (int i = 0; i < 8; ++i) v[k][i] = 0.f;
    }
    int s = 0;
    for (; s + 4 <= ks; s += 4) {
      float4 a[4][NC][2];
#pragma unroll
      for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int k = 0; k < NC; ++k) {
          a[j][k][0] = __ldcg(reinterpret_cast<const float4*>(p[k] + (s + j) * plane));
          a[j][k][1] = __ldcg(reinterpret_cast<const float4*>(p[k] + (s + j) * plane) + 1);
        }
#pragma unroll
      for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int k = 0; k < NC; ++k) {
          v[k][0] += a[j][k][0].x; v[k][1] += a[j][k][0].y; v[k][2] += a[j][k][0].z; v[k][3] += a[j][k][0].w;
          v[k][4] += a[j][k][1].x; v[k][5] += a[j][k][1].y; v[k][6] += a[j][k][1].z; v[k][7] += a[j][k][1].w;
        }
    }
    for (; s < ks; ++s)
#pragma unroll
      for (int k = 0; k < NC; ++k) {
        const float4 a0 = __ldcg(reinterpret_cast<const float4*>(p[k] + s * plane));
        const float4 a1 = __ldcg(reinterpret_cast<const float4*>(p[k] + s * plane) + 1);
        v[k][0] += a0.x; v[k][1] += a0.y; v[k][2] += a0.z; v[k][3] += a0.w;
        v[k][4] += a1.x; v[k][5] += a1.y; v[k][6] += a1.z; v[k][7] += a1.w;
      }
  };
  auto sum8 = [&](int n, float (&v)[8]) {
    const int nn[1] = {n};
    sum_cols(std::integral_constant<int, 1>{}, nn, &v);
  };
  auto sum8x2 = [&](int n0, int n1, float (&v)[8], float (&u)[8]) {
    const int nn[2] = {n0, n1};
    float vu[2][8];
    sum_cols(std::integral_constant<int, 2>{}, nn, vu);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      v[i] = vu[0][i];
      u[i] = vu[1][i];
    }
  };
  float v[8];
  if (e.kind == EPI_SWIGLU_BF16) {
    float u[8];
    sum8x2(c, e.up_off + c, v, u);
    __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(e.out) + c;
    #pragma unroll
    for (int i = 0; i < 8; ++i)
      if (i < mn) o[(size_t)(m0 + i) * e.ldo] = __float2bfloat16_rn(silu(v[i]) * u[i]);
    return;
  }
  if (e.kind == EPI_BF16_ROPE) {
    const int dh = e.head_dim, half = dh >> 1;
    const int hb = (c / dh) * dh, i0 = c - hb;
    __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(e.out) + c;
    if (hb < e.rope_cols) {
      if (i0 >= half) return;  // the pair's first element writes both
      float u[8];
      sum8x2(c, c + half, v, u);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        if (i >= mn) break;
        const int row = m0 + i;
        const int p = __ldg(e.pos + row);
        const bool pos_ok = p >= 0 && p < e.max_pos;
        if (!pos_ok) set_error(err, SP_DEVERR_INDEX);
        const float2 r = __ldg(e.rope + (size_t)(pos_ok ? p : 0) * half + i0);
        o[(size_t)row * e.ldo] = __float2bfloat16_rn(v[i] * r.x - u[i] * r.y);
        o[(size_t)row * e.ldo + half] = __float2bfloat16_rn(u[i] * r.x + v[i] * r.y);
      }
    } else {
      sum8(c, v);
      #pragma unroll
    for (int i = 0; i < 8; ++i)
      if (i < mn) o[(size_t)(m0 + i) * e.ldo] = __float2bfloat16_rn(v[i]);
    }
    return;
  }
  sum8(c, v);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    if (i >= mn) break;
    const int row = m0 + i;
    if (e.kind == EPI_F32) {
      reinterpret_cast<float*>(e.out)[(size_t)row * e.ldo + c] = v[i];
    } else if (e.kind == EPI_F32_ACC) {
      reinterpret_cast<float*>(e.out)[(size_t)row * e.ldo + c] += v[i];
    } else if (e.kind == EPI_GELU_BF16) {
      reinterpret_cast<__nv_bfloat16*>(e.out)[(size_t)row * e.ldo + c] = __float2bfloat16_rn(gelu_erf(v[i]));
    } else if (e.kind == EPI_SCATTER_BF16) {
      const int orow = __ldg(e.row_map + row);
      if (orow < 0) {
        set_error(err, SP_DEVERR_INDEX);
        continue;
      }
      reinterpret_cast<__nv_bfloat16*>(e.out)[(size_t)orow * e.ldo + c] = __float2bfloat16_rn(v[i]);
    } else {
      reinterpret_cast<__nv_bfloat16*>(e.out)[(size_t)row * e.ldo + c] = __float2bfloat16_rn(v[i]);
    }
  }
}

template <int BN, int EPI>
cudaError_t launch_one(const CUtensorMap& A, const CUtensorMap& B, const CUtensorMap& O, const KArgs& a, int grid,
                       cudaStream_t st) {
  using C = Cfg<BN>;
  static bool attr_done = false;  // per (BN, EPI) instantiation
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  cudaError_t le = launch_pdl(gemm_tc_kernel<BN, EPI>, dim3(grid), dim3(192), C::SMEM, st, A, B, O, a);
  if (le != cudaSuccess) return le;
  return cudaGetLastError();
}

template <int BN>
cudaError_t dispatch(const CUtensorMap& A, const CUtensorMap& B, const CUtensorMap& O, const KArgs& a, int grid,
                     cudaStream_t st) {
  switch (a.e.kind) {
    case EPI_BF16: return launch_one<BN, EPI_BF16>(A, B, O, a, grid, st);
    case EPI_BF16_ROPE: return launch_one<BN, EPI_BF16_ROPE>(A, B, O, a, grid, st);
    case EPI_F32: return launch_one<BN, EPI_F32>(A, B, O, a, grid, st);
    case EPI_F32_ACC: return launch_one<BN, EPI_F32_ACC>(A, B, O, a, grid, st);
    case EPI_GELU_BF16: return launch_one<BN, EPI_GELU_BF16>(A, B, O, a, grid, st);
    case EPI_SWIGLU_BF16: return launch_one<BN, EPI_SWIGLU_BF16>(A, B, O, a, grid, st);
    case EPI_SCATTER_BF16: return launch_one<BN, EPI_SCATTER_BF16>(A, B, O, a, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

// K ranges per 128-row weight tile of the weight-streaming GEMM: the split
// that minimises the busiest CTA's K blocks (units t = blockIdx.x + i * grid,
// half a K block of hand-over per unit, ~0.36 us per 16 KB block at an SM's
// share of HBM bandwidth) plus the partial planes' write and read through L2
// (N_acc x 128 bytes per range).  Cached per shape (host-side cost: O(units)).
static int swap_split(int tiles, int KB, int sms, size_t cap_floats, int N_acc) {
  struct Entry { int tiles, KB, sms, N, ks; };
  static thread_local Entry cache[16];
  static thread_local int n_cached = 0;
  for (int i = 0; i < n_cached; ++i)
    if (cache[i].tiles == tiles && cache[i].KB == KB && cache[i].sms == sms && cache[i].N == N_acc)
      return cache[i].ks;
  int best = 1;
  double best_us = 1e30;
  for (int ks = 1; ks <= std::min(16, std::max(1, KB / 2)); ++ks) {
    if ((size_t)ks * N_acc * 32 > cap_floats) break;
    const int U = tiles * ks, G = std::min(U, sms);
    double worst = 0.0;
    for (int c = 0; c < G; ++c) {
      double kb = 0.0;
      for (int u = c; u < U; u += G) {
        const int sp = u % ks;
        kb += (double)((sp + 1) * KB / ks - sp * KB / ks) + 0.5;
      }
      worst = std::max(worst, kb);
    }
    const double us = worst * 0.364 + (double)ks * N_acc * 128.0 / 8.0e6;
    if (us < best_us) {
      best_us = us;
      best = ks;
    }
  }
  if (n_cached < 16) cache[n_cached++] = Entry{tiles, KB, sms, N_acc, best};
  return best;
}

// Tile width of the CTA-pair variant for a GEMM, or 0 for the single-CTA one.
// Pairs with 256-wide tiles wherever M reaches a pair tile: measured on the
// 7B-dims prefill they beat the single-CTA kernel on every GEMM, while 128-wide
// pair tiles lose (the MMA issue per stage no longer hides behind the MMA).
int gemm_pair_policy(int M_cap, int N_acc, int kind) {
  (void)kind;
  if (M_cap < 2 * BM) return 0;
  return N_acc % 256 == 0 ? 256 : 0;
}

size_t gemm_scratch_bytes() {
  const size_t slots = (size_t)(device_sm_count() / 2);
  return slots * kSlotFloats * sizeof(float) + slots * 8 * sizeof(int) + 16 * sizeof(int);
}

GemmScratch gemm_scratch_at(void* p) {
  GemmScratch g;
  if (!p) return g;
  g.slots = device_sm_count() / 2;
  g.part = static_cast<float*>(p);
  g.flags = reinterpret_cast<int*>(g.part + (size_t)g.slots * kSlotFloats);
  g.attn_sched = g.flags + (size_t)g.slots * 8;
  return g;
}

size_t gemm_splitk_floats(int max_n_acc) {
  // split count <= ceil(SMs / tiles) with tiles >= N / 256 and <= 16: planes x N_acc
  // stays below (SMs + N / 128) x 256 per row, 128 rows per plane at most
  const size_t per_row = ((size_t)device_sm_count() + (size_t)max_n_acc / 128 + 1) * 256;
  return per_row * BM;
}

cudaError_t gemm_scratch_clear(const GemmScratch& g, cudaStream_t st) {
  if (!g.flags) return cudaSuccess;
  return cudaMemsetAsync(g.flags, 0, (size_t)g.slots * 8 * sizeof(int) + 16 * sizeof(int), st);
}

bool make_gemm_b(GemmB* b, const void* w, int N, int K, std::string* msg) {
  b->N = N;
  b->K = K;
  return encode_tmap_bf16(&b->map128, w, N, K, 64, msg) &&
         encode_tmap_bf16(&b->map256, w, N, K, 128, msg);
}

cudaError_t gemm_swap_partials(const CUtensorMap& A16, int M_cap, const GemmB& B, int N_acc, int* err,
                               cudaStream_t st, const GemmScratch& sk, int* ks_out) {
  const int sms = device_sm_count();
  if (!sk.splitk || M_cap < 1 || M_cap > 32 || N_acc % BM != 0 || B.K % BK != 0)
    return cudaErrorNotSupported;
  const int tiles = N_acc / BM, KB = B.K / BK;
  const int ks = swap_split(tiles, KB, sms, sk.splitk_floats, N_acc);
  if ((size_t)ks * N_acc * 32 > sk.splitk_floats) return cudaErrorNotSupported;
  CUtensorMap tmP;
  if (!encode_tmap_2d(&tmP, sk.splitk, true, (uint64_t)ks * N_acc, 32, 32, 32, nullptr)) return cudaErrorInvalidValue;
  KArgs a;
  a.M_cap = N_acc;
  a.M_dev = nullptr;
  a.N_acc = 32;
  a.K = B.K;
  a.e = GemmEpi();
  a.e.kind = EPI_F32;
  a.err = err;
  a.a_seg = 0;
  a.a_rows = nullptr;
  a.a_map = 0;
  a.ksplit = ks;
  a.m_pad = N_acc;
  a.swiglu_b = 0;
  a.sk_part = nullptr;
  a.sk_flags = nullptr;
  const int grid = std::max(1, std::min(tiles * ks, sms));
  prof_begin_launch(st);
  const cudaError_t r = launch_one<32, EPI_F32>(B.map256, A16, tmP, a, grid, st);
  prof_end_launch(st, SP_K_GEMM, 2.0 * (double)M_cap * (double)N_acc * (double)B.K, 0.0);
  if (r != cudaSuccess) return r;
  *ks_out = ks;
  return cudaGetLastError();
}

cudaError_t gemm_bf16(const CUtensorMap& A, int M_cap, const int* M_dev, const GemmB& B, int N_acc,
                      const GemmEpi& e, int* err, cudaStream_t st, const GemmScratch* sk,
                      const GemmASplit* as, const CUtensorMap* A16, const int* a_rows) {
  if (M_cap <= 0) return cudaSuccess;
  const int sms = device_sm_count();
  if (a_rows) A16 = nullptr;  // gathered A rows: not the weight-streaming form (M <= 32 rows)
  // Weight streaming for M <= 32 rows (generation steps): the weights are the
  // MMA's 128-row operand and the activations its 32 columns (C^T = B A^T),
  // each 128-row weight tile's K split into ranges over the SMs; the fp32
  // partials [range][N_acc][32] are summed, with the fused epilogue, by one
  // transposed reduce pass.
  if (A16 && sk) {
    int ks = 0;
    const cudaError_t r = gemm_swap_partials(*A16, M_cap, B, N_acc, err, st, *sk, &ks);
    if (r == cudaSuccess) {
      const int cols = e.kind == EPI_SWIGLU_BF16 ? N_acc / 2 : N_acc;
      prof_begin_launch(st);
      const cudaError_t rr = launch_pdl(splitk_reduce_t_kernel, dim3((cols * 4 + 255) / 256), dim3(256), 0, st,
                                        sk->splitk, ks, N_acc, M_cap, M_dev, cols, e, err);
      prof_end_launch(st, SP_K_MISC, 0.0, 4.0 * ks * (double)N_acc * 32);
      if (rr != cudaSuccess) return rr;
      return cudaGetLastError();
    }
    if (r != cudaErrorNotSupported) return r;
  }
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
  a.sk_part = nullptr;
  a.sk_flags = nullptr;
  a.a_seg = 0;
  a.a_rows = nullptr;
  a.a_map = 0;
  a.ksplit = 1;
  a.m_pad = 0;
  a.swiglu_b = 0;
  if (as && as->seg > 0) {
    if (as->seg % BK != 0 || B.K > 8 * as->seg) return cudaErrorInvalidValue;
    a.a_seg = as->seg;
    a.a_map = as->map;
  }
  a.a_rows = a_rows;
  // output map for the TMA epilogue (box 32 rows x 128 bytes); the row-scatter
  // epilogue stores directly and needs none
  CUtensorMap tmO;
  std::memset(&tmO, 0, sizeof(tmO));
  if (e.kind != EPI_SCATTER_BF16) {
    const bool f32 = e.kind == EPI_F32 || e.kind == EPI_F32_ACC;
    if (!encode_tmap_2d(&tmO, e.out, f32, (uint64_t)M_cap, (uint64_t)e.ldo, f32 ? 32 : 64, 32, nullptr))
      return cudaErrorInvalidValue;
  }
  cudaError_t r;
  const int pair_bn = gemm_pair_policy(M_cap, N_acc, e.kind);
  if (pair_bn) {
    const int mp = (M_cap + 2 * BM - 1) / (2 * BM);
    const int tiles = mp * (N_acc / pair_bn);
    int slots = 0;
    if (sk && sk->part && sk->flags) {
      a.sk_part = sk->part;
      a.sk_flags = sk->flags;
      slots = sk->slots;
    }
    prof_begin_launch(st);
    r = pair_bn == 256 ? dispatch_pair<256>(A, B.map256, tmO, a, tiles, slots, st)
                       : dispatch_pair<128>(A, B.map128, tmO, a, tiles, slots, st);
    prof_end_launch(st, SP_K_GEMM, 2.0 * (double)M_cap * (double)N_acc * (double)B.K, 0.0);
    return r;
  }
  const int bn = use256 ? 256 : 128;
  const int tiles = mt * (N_acc / bn);
  double flops = 2.0 * (double)M_cap * (double)N_acc * (double)B.K;
  // Small M (<= 128 rows: generation steps, one short sequence): too few tiles
  // to stream the weights with every SM; split K into ranges over the idle SMs,
  // fp32 partials to the caller's scratch, then one reduce + epilogue pass.
  const int KB = B.K / BK;
  if (sk && sk->splitk && M_cap <= BM && tiles < sms && KB >= 8) {
    int kspl = std::min(std::min((sms + tiles - 1) / tiles, KB / 4), 16);
    const int m_pad = (M_cap + 31) / 32 * 32;
    while (kspl > 1 && (size_t)kspl * m_pad * N_acc > sk->splitk_floats) --kspl;
    if (kspl > 1) {
      CUtensorMap tmP;
      if (!encode_tmap_2d(&tmP, sk->splitk, true, (uint64_t)kspl * m_pad, (uint64_t)N_acc, 32, 32, nullptr))
        return cudaErrorInvalidValue;
      KArgs ap = a;
      ap.e.kind = EPI_F32;
      ap.ksplit = kspl;
      ap.m_pad = m_pad;
      ap.swiglu_b = e.kind == EPI_SWIGLU_BF16 ? 1 : 0;
      const int grid = std::max(1, std::min(tiles * kspl, sms));
      prof_begin_launch(st);
      r = use256 ? launch_one<256, EPI_F32>(A, B.map256, tmP, ap, grid, st)
                 : launch_one<128, EPI_F32>(A, B.map128, tmP, ap, grid, st);
      prof_end_launch(st, SP_K_GEMM, flops, 0.0);
      if (r != cudaSuccess) return r;
      const int cols = e.kind == EPI_SWIGLU_BF16 ? N_acc / 2 : N_acc;
      dim3 rg((cols + 255) / 256, M_cap);
      prof_begin_launch(st);
      cudaError_t re = launch_pdl(splitk_reduce_kernel, dim3(rg), dim3(256), 0, st, sk->splitk, kspl, m_pad, M_cap,
                                  M_dev, N_acc, bn, e, err);
      if (re != cudaSuccess) return re;
      prof_end_launch(st, SP_K_MISC, 0.0, 4.0 * kspl * (double)m_pad * N_acc);
      return cudaGetLastError();
    }
  }
  const int grid = std::max(1, std::min(tiles, sms));
  prof_begin_launch(st);
  r = use256 ? dispatch<256>(A, B.map256, tmO, a, grid, st)
             : dispatch<128>(A, B.map128, tmO, a, grid, st);
  prof_end_launch(st, SP_K_GEMM, flops, 0.0);
  return r;
}

}  // namespace sp
