// Variable-length attention over packed sequences (cu_seqlens), causal for the
// LM prefill and bidirectional for the selector's cross-modal encoder (Eq. 3,
// Table 7(a)); grouped-query heads map query head i to kv head i / (Hq / Hkv).
// One tcgen05 kernel (below) serves both, head dims 64 and 128.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

// ===========================================================================
// Persistent tcgen05 flash attention.  One CTA per SM walks a static list of
// work items, an item being 128 query rows (one tile) of one head of one
// sequence, longest tiles first.
//
//   warp 0      TMA: the Q tile once per item, then per 128-key block the K
//               block into a three-slot ring and the V block into a two-slot
//               ring
//   warp 1      issues the scores S = Q K^T (M 128, N 128, both K-major from
//               shared memory) into one of three S / P buffers in TMEM; it also
//               allocates the 512 TMEM columns
//   warp 2      issues O += P V (P read from Tensor Memory where the softmax
//               wrote it over its S, V an MN-major operand straight from its
//               TMA block)
//   warps 4-7   softmax of key columns 0-63 of every block, warps 8-11 of
//               columns 64-127: one thread per (query row = TMEM lane, half);
//               the two halves of a row exchange their block maxima through
//               shared memory (an mbarrier per pair of warps, bounded waits),
//               so both keep the same running max.  Running max / sum in the exp2 domain,
//               P as bf16 back over S, O rescaled in TMEM only when the running
//               max grows by more than 2^8 (lazy rescale: O and the sum l share
//               the stale max, so the result is exact), final O / l to global
//               (each half of the warps stores half of the head dims).
// Three S / P buffers let the scores run up to two blocks ahead of the
// softmax; the scores of block j + 3 reuse block j's buffer only once O += P V
// of block j has completed.  Each issuing thread waits once per block: the K
// barrier of block j counts the TMA's arrival (with K's bytes) and the commit
// of O += P V of block j - 3; the P barrier counts the eight softmax warps and
// the TMA's arrival with V's bytes.  A K slot is free once the scores that read
// it are complete, a V slot once O += P V is: no "empty" barriers.
// TMEM columns: S / P buffer b at [128 b, 128 b + 128) (P: 64 columns of bf16
// pairs over the first half of S), O at [384, 384 + DH).
// Keys past the sequence get P = 0; their V rows must be finite (the caller
// keeps the rows past the packed length zero, or the tensor map ends there).
namespace fa {

constexpr int BQ = 128, BKV = 128, NTHR = 384, NSB = 3, NVS = 2;
constexpr float kRescaleLog2 = 8.f;  // rescale O once the max moved by more than this (log2 units)

template <int DH>
struct Cfg {
  static constexpr uint32_t BOX = 128 * 128;               // 128 rows x 64 bf16 (one 128-byte swizzle box)
  static constexpr uint32_t TILE = DH / 64 * BOX;          // a Q tile or a K / V block
  static constexpr uint32_t OFF_Q = 0;
  static constexpr uint32_t OFF_K = TILE;                  // [NSB]
  static constexpr uint32_t OFF_V = OFF_K + NSB * TILE;    // [NVS]
  static constexpr uint32_t OFF_X = OFF_V + NVS * TILE;    // softmax exchange: [2 blocks][2 halves][128] floats
  static constexpr uint32_t OFF_BAR = OFF_X + 6 * 128 * 4;  //   then the row sums [2 halves][128]
  static constexpr size_t SMEM_USED = 1024 + OFF_BAR + 512;
  // a CTA holds all 512 TMEM columns: ask for more than half of the shared
  // memory so that a second CTA is never co-resident (it would only wait)
  static constexpr size_t SMEM = SMEM_USED > 120 * 1024 ? SMEM_USED : 120 * 1024;
  static constexpr uint32_t T_O = 384;
};

// Barriers; X + s for the slot / buffer s of a block.  XB + 2 q + (block & 1)
// and XL + q: the exchanges between the two softmax warps of lane quadrant q.
enum Bar {
  Q_FULL = 0, Q_EMPTY = 1, K_FULL = 2, S_FULL = 5, P_FULL = 8, PV_DONE = 11, O_FULL = 14, O_EMPTY = 15,
  MMA_DONE = 16, XB = 18, XL = 26, N_BARS = 30
};

SP_DEVINL float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

SP_DEVINL float max3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// The two softmax warps of a lane quadrant publish their values for each other:
// the warp's writes, then one arrival (count 2: both warps); a bounded wait.
SP_DEVINL bool pair_exchange(uint64_t* b, uint32_t parity, int* err) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(b);
  return mbar_wait_warp(b, parity, err);
}

struct Item {
  int s0, len, q0, h, kvh, nkv;
};

// Work item `it` of the static list: query tiles from the last (the most key
// blocks under a causal mask) to the first; within a tile index, sequence-major,
// then head.  Returns false for tiles past the sequence's end.
SP_DEVINL bool item_at(int it, const int* __restrict__ cu, int B, int Hq, int n_tiles, int Hkv, bool causal,
                       Item& I) {
  const int per_tile = B * Hq;
  const int tile = n_tiles - 1 - it / per_tile;
  const int rem = it - (it / per_tile) * per_tile;
  const int b = rem / Hq;
  I.h = rem - b * Hq;
  I.s0 = __ldg(cu + b);
  I.len = __ldg(cu + b + 1) - I.s0;
  I.q0 = tile * BQ;
  if (I.q0 >= I.len) return false;
  I.kvh = I.h / (Hq / Hkv);
  const int kend = causal ? min(I.len, I.q0 + BQ) : I.len;
  I.nkv = (kend + BKV - 1) / BKV;
  return true;
}

template <int DH>
__global__ void __launch_bounds__(NTHR, 1)
attn_fa_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKV,
               __nv_bfloat16* __restrict__ out, const int* __restrict__ cu, int B, int Hq, int Hkv, int n_tiles,
               int ld_out, int causal_i, float scale_log2, int* err) {
  using C = Cfg<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + C::OFF_BAR);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + N_BARS);
  float* xchg = reinterpret_cast<float*>(sm + C::OFF_X);
  const bool causal = causal_i != 0;
  const int n_items = n_tiles * B * Hq;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < N_BARS; ++i) {
      uint32_t n = 1;
      if (i >= K_FULL && i < K_FULL + NSB) n = 2;   // TMA + O += P V of block - 3
      if (i >= P_FULL && i < P_FULL + NSB) n = 9;   // 8 softmax warps + TMA (V)
      if (i == O_EMPTY) n = 8;
      if (i >= XB) n = 2;                           // the two softmax warps of a quadrant
      mbar_init(&bar[i], n);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tslot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  pdl_wait();  // programmatic launch: the previous kernel's outputs are visible from here
  pdl_trigger();

  if (warp == 0) {
    // ------------------------------------------------------------ TMA
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmKV);
      uint32_t g = 0, nitem = 0;
      bool ok = true;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
        Item I;
        if (!item_at(it, cu, B, Hq, n_tiles, Hkv, causal, I)) continue;
        if (!mbar_wait(&bar[Q_EMPTY], (nitem & 1) ^ 1u, err)) break;
        mbar_arrive_expect_tx(&bar[Q_FULL], C::TILE);
#pragma unroll
        for (int bx = 0; bx < DH / 64; ++bx)
          tma_load_2d(sm + C::OFF_Q + bx * C::BOX, &tmQ, &bar[Q_FULL], I.h * DH + bx * 64, I.s0 + I.q0);
        const int kcol = (Hq + I.kvh) * DH, vcol = (Hq + Hkv + I.kvh) * DH;
        for (int j = 0; j < I.nkv; ++j, ++g) {
          const uint32_t ks = g % NSB, kph = (g / NSB) & 1;
          // K slot ks last held block g - 3: free once its scores are complete
          if (g >= NSB && !mbar_wait(&bar[S_FULL + ks], kph ^ 1u, err)) { ok = false; break; }
          mbar_arrive_expect_tx(&bar[K_FULL + ks], C::TILE);
          if (g < NSB) mbar_arrive(&bar[K_FULL + ks]);  // (no O += P V of block g - 3 arrives)
#pragma unroll
          for (int bx = 0; bx < DH / 64; ++bx)
            tma_load_2d(sm + C::OFF_K + ks * C::TILE + bx * C::BOX, &tmKV, &bar[K_FULL + ks], kcol + bx * 64,
                        I.s0 + j * BKV);
          // V slot g % 2 last held block g - 2: free once its O += P V is complete
          if (g >= NVS) {
            const uint32_t pg = g - NVS;
            if (!mbar_wait(&bar[PV_DONE + pg % NSB], (pg / NSB) & 1, err)) { ok = false; ++g; break; }
          }
          mbar_arrive_expect_tx(&bar[P_FULL + ks], C::TILE);
#pragma unroll
          for (int bx = 0; bx < DH / 64; ++bx)
            tma_load_2d(sm + C::OFF_V + (g % NVS) * C::TILE + bx * C::BOX, &tmKV, &bar[P_FULL + ks],
                        vcol + bx * 64, I.s0 + j * BKV);
        }
        ++nitem;
      }
      // every copy lands before the CTA may exit (bounded waits; normally
      // the consumers have waited for all of them already)
      if (nitem > 0) mbar_wait(&bar[Q_FULL], (nitem - 1) & 1, err);
      for (uint32_t gg = g >= NSB ? g - NSB : 0; gg < g; ++gg) {
        mbar_wait(&bar[K_FULL + gg % NSB], (gg / NSB) & 1, err);
        mbar_wait(&bar[P_FULL + gg % NSB], (gg / NSB) & 1, err);  // (V, and the block's P)
      }
    }
  } else if (warp == 1 || warp == 2) {
    // ------------------------------------------------------------ MMA issuers
    // warp 1: the scores; warp 2: O += P V (tcgen05.commit tracks the issuing
    // thread's own MMAs; the two write disjoint TMEM columns)
    if (lane == 0) {
      const bool pv_issuer = warp == 2;
      constexpr uint32_t IDESC_S = umma_idesc_bf16_f32(BQ, BKV);
      constexpr uint32_t IDESC_O = umma_idesc_bf16_f32(BQ, DH) | (1u << 16);  // B (V) MN-major
      // shared-memory descriptors of the slot bases; a K step adds its byte
      // offset / 16 to the address field (it stays below the field's 14 bits)
      const uint64_t dQ = umma_desc_sw128(smem_u32(sm + C::OFF_Q));
      const uint64_t dK = umma_desc_sw128(smem_u32(sm + C::OFF_K));
      const uint64_t dV = umma_desc_sw128_mn(smem_u32(sm + C::OFF_V), C::BOX);
      const uint64_t slot16 = C::TILE >> 4;
      uint32_t g = 0, nitem = 0;
      bool ok = true;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
        Item I;
        if (!item_at(it, cu, B, Hq, n_tiles, Hkv, causal, I)) continue;
        if (!pv_issuer) {
          ok = mbar_wait(&bar[Q_FULL], nitem & 1, err);
          for (int j = 0; ok && j < I.nkv; ++j) {
            const uint32_t gg = g + j, sb = gg % NSB;
            // the K barrier also counts O += P V of block gg - 3, the last reader of buffer sb
            if (!mbar_wait(&bar[K_FULL + sb], (gg / NSB) & 1, err)) { ok = false; break; }
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < DH / 16; ++kk)
              umma_bf16(tmem + sb * BKV, dQ + (((kk >> 2) * C::BOX + (kk & 3) * 32) >> 4),
                        dK + sb * slot16 + (((kk >> 2) * C::BOX + (kk & 3) * 32) >> 4), IDESC_S, kk ? 1u : 0u);
            umma_commit(&bar[S_FULL + sb]);
            if (j + 1 == I.nkv) umma_commit(&bar[Q_EMPTY]);
          }
        } else {
          for (int j = 0; ok && j < I.nkv; ++j) {
            const uint32_t gg = g + j, sb = gg % NSB;
            // P_FULL completes once the softmax wrote P and the block's V landed
            if (!mbar_wait(&bar[P_FULL + sb], (gg / NSB) & 1, err) ||
                (j == 0 && !mbar_wait(&bar[O_EMPTY], (nitem & 1) ^ 1u, err))) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint64_t dVs = dV + (gg % NVS) * slot16;
#pragma unroll
            for (int kk = 0; kk < BKV / 16; ++kk)
              umma_bf16_ta(tmem + C::T_O, tmem + sb * BKV + kk * 8, dVs + ((kk * 2048) >> 4), IDESC_O,
                           (j | kk) ? 1u : 0u);
            umma_commit(&bar[PV_DONE + sb]);
            umma_commit(&bar[K_FULL + sb]);  // (counts toward block gg + 3's K barrier)
            if (j + 1 == I.nkv) umma_commit(&bar[O_FULL]);
          }
        }
        g += I.nkv;
        ++nitem;
      }
      // TMEM stays allocated until every MMA this thread issued is done
      umma_commit(&bar[MMA_DONE + (pv_issuer ? 1 : 0)]);
      mbar_wait(&bar[MMA_DONE + (pv_issuer ? 1 : 0)], 0, err);
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ------------------------------------------------------------ softmax (row = TMEM lane, half of the keys)
    const int half = (warp - 4) >> 2;
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    constexpr int HC = BKV / 2;  // key columns of a half
    float* xmax = xchg;           // [2 blocks][2 halves][128]
    uint32_t g = 0, nitem = 0;
    bool ok = true;
    for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
      Item I;
      if (!item_at(it, cu, B, Hq, n_tiles, Hkv, causal, I)) continue;
      const int qpos = I.q0 + r;  // query position in the sequence
      const int row_lim = qpos >= I.len ? 0 : (causal ? qpos + 1 : I.len);  // keys [0, row_lim) are visible
      float m = -INFINITY, l = 0.f;  // m: running max in log2 units; l: this half's sum
      for (int j = 0; j < I.nkv; ++j, ++g) {
        const uint32_t sb = g % NSB;
        if (!mbar_wait_warp(&bar[S_FULL + sb], (g / NSB) & 1, err)) { ok = false; break; }
        tc_fence_after();
        float v[HC];
        tmem_ld_32x32b_x32(trow + sb * BKV + half * HC, *reinterpret_cast<float(*)[32]>(v));
        tmem_ld_32x32b_x32(trow + sb * BKV + half * HC + 32, *reinterpret_cast<float(*)[32]>(v + 32));
        tmem_ld_wait();
        const int lim = row_lim - j * BKV - half * HC;
        if (lim < HC) {
#pragma unroll
          for (int c = 0; c < HC; ++c) v[c] = c < lim ? v[c] : -INFINITY;
        }
        float mx[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mx[e] = max3(v[e], v[e + 8], v[e + 16]);
#pragma unroll
        for (int e = 0; e < 8; ++e) mx[e] = max3(mx[e], v[e + 24], v[e + 32]);
#pragma unroll
        for (int e = 0; e < 8; ++e) mx[e] = max3(mx[e], v[e + 40], v[e + 48]);
#pragma unroll
        for (int e = 0; e < 8; ++e) mx[e] = fmaxf(mx[e], v[e + 56]);
        float mh = max3(max3(mx[0], mx[1], mx[2]), max3(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7]));
        // the block max of the whole row: exchange with the other half (double-buffered by block)
        float* xb = xmax + (g & 1) * 256;
        xb[half * 128 + r] = mh;
        if (!pair_exchange(&bar[XB + 2 * quad + (g & 1)], (g >> 1) & 1, err)) { ok = false; break; }
        const float mb = fmaxf(mh, xb[(half ^ 1) * 128 + r]) * scale_log2;
        // stale-max rule: move m (and rescale O and l) only when the block max exceeds it by > 2^8
        float corr = 1.f;
        bool moved = false;
        if (mb > m + kRescaleLog2 || (m == -INFINITY && mb > -INFINITY)) {
          corr = m == -INFINITY ? 0.f : ex2(m - mb);
          moved = m != -INFINITY;
          m = mb;
        }
        const float nm = m == -INFINITY ? 0.f : -m;
        float ls[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) ls[e] = 0.f;
        float pk[HC / 2];  // bf16 pairs, bit-cast for tcgen05.st
#pragma unroll
        for (int e = 0; e < HC / 2; ++e) {
          const float p0 = ex2(fmaf(v[2 * e], scale_log2, nm)), p1 = ex2(fmaf(v[2 * e + 1], scale_log2, nm));
          ls[(2 * e) & 7] += p0;
          ls[(2 * e + 1) & 7] += p1;
          pk[e] = __uint_as_float(pack_bf16x2(p0, p1));
        }
        l = l * corr + ((ls[0] + ls[1]) + (ls[2] + ls[3])) + ((ls[4] + ls[5]) + (ls[6] + ls[7]));
        if (__any_sync(0xffffffffu, moved)) {
          // O += P V of the previous block must be done with O before it is rescaled;
          // each half rescales its half of the head dims
          const uint32_t pg = g - 1;
          if (!mbar_wait_warp(&bar[PV_DONE + pg % NSB], (pg / NSB) & 1, err)) { ok = false; break; }
          tc_fence_after();
          float o[32];
#pragma unroll 1
          for (int c = half * (DH / 2); c < (half + 1) * (DH / 2); c += 32) {
            tmem_ld_32x32b_x32(trow + C::T_O + c, o);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] *= corr;
            tmem_st_32x32b_x32(trow + C::T_O + c, o);
          }
        }
        tmem_st_32x32b_x32(trow + sb * BKV + half * (HC / 2), pk);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar[P_FULL + sb]);
      }
      if (!ok) break;
      // ---- O / l to global: the row's sum is the two halves' sums
      float* xl = xmax + 512;  // [2 halves][128]
      xl[half * 128 + r] = l;
      if (!pair_exchange(&bar[XL + quad], nitem & 1, err)) { ok = false; break; }
      const float lt = l + xl[(half ^ 1) * 128 + r];
      if (!mbar_wait_warp(&bar[O_FULL], nitem & 1, err)) { ok = false; break; }
      tc_fence_after();
      const float inv = lt > 0.f ? 1.f / lt : 0.f;
      const bool store = qpos < I.len;
      __nv_bfloat16* dst = out + (size_t)(I.s0 + qpos) * ld_out + I.h * DH;
      float o[32];
#pragma unroll 1
      for (int c = half * (DH / 2); c < (half + 1) * (DH / 2); c += 32) {
        tmem_ld_32x32b_x32(trow + C::T_O + c, o);
        tmem_ld_wait();
        if (store) {
          uint4* d4 = reinterpret_cast<uint4*>(dst + c);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint4 u;
            u.x = pack_bf16x2(o[8 * q + 0] * inv, o[8 * q + 1] * inv);
            u.y = pack_bf16x2(o[8 * q + 2] * inv, o[8 * q + 3] * inv);
            u.z = pack_bf16x2(o[8 * q + 4] * inv, o[8 * q + 5] * inv);
            u.w = pack_bf16x2(o[8 * q + 6] * inv, o[8 * q + 7] * inv);
            d4[q] = u;
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar[O_EMPTY]);
      ++nitem;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

}  // namespace fa
}  // namespace

template <int DH>
cudaError_t launch_attn_fa(const void* qkv, void* out, const int* cu, int B, int max_len, int rows_cap, int Hq,
                           int Hkv, bool causal, float scale_log2, int* err, cudaStream_t st) {
  using C = fa::Cfg<DH>;
  static bool attr = false;
  if (!attr) {
    cudaError_t r = cudaFuncSetAttribute(fa::attn_fa_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::SMEM);
    if (r != cudaSuccess) return r;
    attr = true;
  }
  if (Hkv <= 0 || Hq % Hkv != 0) return cudaErrorInvalidValue;
  const int ld_qkv = (Hq + 2 * Hkv) * DH;
  CUtensorMap tq, tkv;
  if (!encode_tmap_2d(&tq, qkv, false, (uint64_t)rows_cap, (uint64_t)ld_qkv, 64, fa::BQ, nullptr) ||
      !encode_tmap_2d(&tkv, qkv, false, (uint64_t)rows_cap, (uint64_t)ld_qkv, 64, fa::BKV, nullptr))
    return cudaErrorInvalidValue;
  const int n_tiles = (max_len + fa::BQ - 1) / fa::BQ;
  const long n_items = (long)n_tiles * B * Hq;
  const int grid = (int)std::min<long>(n_items, (long)device_sm_count());
  return launch_pdl(fa::attn_fa_kernel<DH>, dim3(grid), dim3(fa::NTHR), C::SMEM, st, tq, tkv,
                    reinterpret_cast<__nv_bfloat16*>(out), cu, B, Hq, Hkv, n_tiles, Hq * DH, causal ? 1 : 0,
                    scale_log2, err);
}

cudaError_t attention_varlen(const void* qkv, void* out, const int* cu_seqlens, int B,
                             int max_seqlen_cap, int rows_cap, int Hq, int Hkv, int dh, bool causal,
                             int* err, cudaStream_t st) {
  if (B <= 0 || max_seqlen_cap <= 0 || rows_cap <= 0) return cudaSuccess;
  const float sl2 = 1.4426950408889634f / sqrtf((float)dh);
  prof_begin_launch(st);
  cudaError_t r = dh == 128 ? launch_attn_fa<128>(qkv, out, cu_seqlens, B, max_seqlen_cap, rows_cap, Hq, Hkv, causal,
                                                  sl2, err, st)
                : dh == 64  ? launch_attn_fa<64>(qkv, out, cu_seqlens, B, max_seqlen_cap, rows_cap, Hq, Hkv, causal,
                                                 sl2, err, st)
                            : cudaErrorInvalidValue;
  prof_end_launch(st, SP_K_ATTN, 0.0, 0.0);
  return r;
}

}  // namespace sp
