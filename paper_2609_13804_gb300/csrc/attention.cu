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
// work items; an item is 128 query rows (one tile) of one sequence for a PAIR
// of query heads (2p, 2p + 1).  The two heads see the same keys positions and
// the same mask, so their pipelines advance in lockstep and the tensor pipe
// alternates between them: while one head's softmax runs, the other head's
// S = Q K^T or O += P V keeps the tensor cores busy.
//
//   warp 0      TMA: per head its Q tile once per item, then per 128-key block
//               its K and V blocks (one buffer each per head; the next block's
//               load starts as soon as the MMA that read the buffer is done)
//   warp 1      TMEM allocation (all 512 columns); one thread issues, per key
//               block: S_0 = Q_0 K_0^T, S_1 = Q_1 K_1^T (M 128, N 128, both
//               K-major from shared memory), then O_0 += P_0 V_0 and
//               O_1 += P_1 V_1 with P read from Tensor Memory (where the
//               softmax wrote it over its S) and V an MN-major operand straight
//               from its TMA block.  Before S_t overwrites P_t, the previous
//               O_t += P_t V_t must have completed (its commit is waited on).
//   warps 2-3   idle
//   warps 4-7   softmax of head 0, warps 8-11 of head 1: one thread per query
//               row (= TMEM lane): S row from TMEM, mask (causal diagonal
//               block, sequence tail), running max / sum in the exp2 domain, P
//               as bf16 back over S, O rescaled in TMEM only when the running
//               max grows by more than 2^8 (lazy rescale: O and the sum l share
//               the stale max, so the result is exact), final O / l to global.
// TMEM columns: S / P of head t at [128 t, 128 t + 128) (P: 64 columns of
// bf16 pairs over the first half of S), O of head t at [256 + DH t, + DH).
// Keys past the sequence get P = 0; their V rows must be finite (the caller
// keeps the rows past the packed length zero, or the tensor map ends there).
namespace fa {

constexpr int BQ = 128, BKV = 128, NTHR = 384;
constexpr float kRescaleLog2 = 8.f;  // rescale O once the max moved by more than this (log2 units)

template <int DH>
struct Cfg {
  static constexpr uint32_t BOX_BYTES = 128 * 128;      // 128 rows x 64 bf16 (one 128-byte swizzle box)
  static constexpr uint32_t TILE_BYTES = DH / 64 * BOX_BYTES;  // a Q tile or a K / V block of one head
  static constexpr uint32_t OFF_Q = 0;                   // [2 heads]
  static constexpr uint32_t OFF_K = 2 * TILE_BYTES;      // [2 heads]
  static constexpr uint32_t OFF_V = 4 * TILE_BYTES;      // [2 heads]
  static constexpr uint32_t OFF_BAR = 6 * TILE_BYTES;
  static constexpr size_t SMEM_USED = 1024 + OFF_BAR + 256;
  // a CTA holds all 512 TMEM columns: ask for more than half of the shared
  // memory so that a second CTA is never co-resident (it would only wait)
  static constexpr size_t SMEM = SMEM_USED > 120 * 1024 ? SMEM_USED : 120 * 1024;
  static constexpr uint32_t T_O = 256;
};

// Barriers, per head t: index base + t.
enum Bar {
  Q_FULL = 0, Q_EMPTY = 2, K_FULL = 4, K_EMPTY = 6, V_FULL = 8, V_EMPTY = 10,
  S_FULL = 12, P_FULL = 14, PV_DONE = 16, O_FULL = 18, O_EMPTY = 20, MMA_DONE = 22, N_BARS = 23
};

SP_DEVINL float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

struct Item {
  int s0, len, q0, h0, h1, kvh0, kvh1, nkv;
};

// Work item `it` of the static list: query tiles from the last (the most key
// blocks under a causal mask) to the first; within a tile index, sequence-major,
// then head pair.  Returns false for tiles past the sequence's end.
SP_DEVINL bool item_at(int it, const int* __restrict__ cu, int B, int HP, int n_tiles, int Hq, int Hkv, bool causal,
                       Item& I) {
  const int per_tile = B * HP;
  const int tile = n_tiles - 1 - it / per_tile;
  const int rem = it - (it / per_tile) * per_tile;
  const int b = rem / HP, hp = rem - (rem / HP) * HP;
  I.s0 = __ldg(cu + b);
  I.len = __ldg(cu + b + 1) - I.s0;
  I.q0 = tile * BQ;
  if (I.q0 >= I.len) return false;
  const int grp = Hq / Hkv;
  I.h0 = 2 * hp;
  I.h1 = min(2 * hp + 1, Hq - 1);  // odd head count: the last pair computes its head twice, stores it once
  I.kvh0 = I.h0 / grp;
  I.kvh1 = I.h1 / grp;
  const int kend = causal ? min(I.len, I.q0 + BQ) : I.len;
  I.nkv = (kend + BKV - 1) / BKV;
  return true;
}

template <int DH>
__global__ void __launch_bounds__(NTHR, 1)
attn_fa_kernel(const __grid_constant__ CUtensorMap tm, __nv_bfloat16* __restrict__ out, const int* __restrict__ cu,
               int B, int Hq, int Hkv, int n_tiles, int ld_out, int causal_i, float scale_log2, int* err) {
  using C = Cfg<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + C::OFF_BAR);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + N_BARS);
  const bool causal = causal_i != 0;
  const int HP = (Hq + 1) / 2;
  const int n_items = n_tiles * B * HP;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < N_BARS; ++i) mbar_init(&bar[i], (i == P_FULL || i == P_FULL + 1 || i == O_EMPTY || i == O_EMPTY + 1) ? 4 : 1);
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
      tma_prefetch_desc(&tm);
      uint32_t g = 0, nitem = 0;
      bool ok = true;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
        Item I;
        if (!item_at(it, cu, B, HP, n_tiles, Hq, Hkv, causal, I)) continue;
#pragma unroll
        for (int t = 0; t < 2; ++t) {
          if (!mbar_wait(&bar[Q_EMPTY + t], (nitem & 1) ^ 1u, err)) { ok = false; break; }
          mbar_arrive_expect_tx(&bar[Q_FULL + t], C::TILE_BYTES);
          uint8_t* dst = sm + C::OFF_Q + t * C::TILE_BYTES;
          const int col = (t ? I.h1 : I.h0) * DH;
#pragma unroll
          for (int bx = 0; bx < DH / 64; ++bx)
            tma_load_2d(dst + bx * C::BOX_BYTES, &tm, &bar[Q_FULL + t], col + bx * 64, I.s0 + I.q0);
        }
        for (int j = 0; ok && j < I.nkv; ++j, ++g) {
          const uint32_t pe = (g & 1) ^ 1u;
#pragma unroll
          for (int kv = 0; kv < 2; ++kv) {  // K of both heads, then V of both heads
#pragma unroll
            for (int t = 0; t < 2; ++t) {
              const int e_bar = (kv ? V_EMPTY : K_EMPTY) + t, f_bar = (kv ? V_FULL : K_FULL) + t;
              if (!mbar_wait(&bar[e_bar], pe, err)) { ok = false; break; }
              mbar_arrive_expect_tx(&bar[f_bar], C::TILE_BYTES);
              uint8_t* dst = sm + (kv ? C::OFF_V : C::OFF_K) + t * C::TILE_BYTES;
              const int kvh = t ? I.kvh1 : I.kvh0;
              const int col = (kv ? Hq + Hkv + kvh : Hq + kvh) * DH;
#pragma unroll
              for (int bx = 0; bx < DH / 64; ++bx)
                tma_load_2d(dst + bx * C::BOX_BYTES, &tm, &bar[f_bar], col + bx * 64, I.s0 + j * BKV);
            }
            if (!ok) break;
          }
        }
        ++nitem;
      }
      // every copy lands before the CTA may exit (bounded waits; normally
      // the consumers have waited for all of them already)
      if (nitem > 0)
        for (int t = 0; t < 2; ++t) mbar_wait(&bar[Q_FULL + t], (nitem - 1) & 1, err);
      if (g > 0)
        for (int t = 0; t < 2; ++t) {
          mbar_wait(&bar[K_FULL + t], (g - 1) & 1, err);
          mbar_wait(&bar[V_FULL + t], (g - 1) & 1, err);
        }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t IDESC_S = umma_idesc_bf16_f32(BQ, BKV);
      constexpr uint32_t IDESC_O = umma_idesc_bf16_f32(BQ, DH) | (1u << 16);  // B (V) MN-major
      uint32_t g = 0, nitem = 0;
      bool ok = true;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
        Item I;
        if (!item_at(it, cu, B, HP, n_tiles, Hq, Hkv, causal, I)) continue;
        for (int t = 0; t < 2 && ok; ++t) ok = mbar_wait(&bar[Q_FULL + t], nitem & 1, err);
        for (int j = 0; ok && j < I.nkv; ++j, ++g) {
          const uint32_t ph = g & 1;
          const bool last = j == I.nkv - 1;
#pragma unroll
          for (int t = 0; t < 2; ++t) {
            // S_t overwrites P_t: the previous O_t += P_t V_t must be complete
            if (!mbar_wait(&bar[K_FULL + t], ph, err) || (g > 0 && !mbar_wait(&bar[PV_DONE + t], (g - 1) & 1, err))) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a0 = smem_u32(sm + C::OFF_Q + t * C::TILE_BYTES);
            const uint32_t b0 = smem_u32(sm + C::OFF_K + t * C::TILE_BYTES);
#pragma unroll
            for (int kk = 0; kk < DH / 16; ++kk) {
              const uint32_t o = (kk >> 2) * C::BOX_BYTES + (kk & 3) * 32;
              umma_bf16(tmem + t * BKV, umma_desc_sw128(a0 + o), umma_desc_sw128(b0 + o), IDESC_S, kk ? 1u : 0u);
            }
            umma_commit(&bar[S_FULL + t]);
            umma_commit(&bar[K_EMPTY + t]);
            if (last) umma_commit(&bar[Q_EMPTY + t]);
          }
          if (!ok) break;
#pragma unroll
          for (int t = 0; t < 2; ++t) {
            if (!mbar_wait(&bar[V_FULL + t], ph, err) || !mbar_wait(&bar[P_FULL + t], ph, err) ||
                (j == 0 && !mbar_wait(&bar[O_EMPTY + t], (nitem & 1) ^ 1u, err))) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t bv = smem_u32(sm + C::OFF_V + t * C::TILE_BYTES);
#pragma unroll
            for (int kk = 0; kk < BKV / 16; ++kk)
              umma_bf16_ta(tmem + C::T_O + t * DH, tmem + t * BKV + kk * 8,
                           umma_desc_sw128_mn(bv + kk * 2048, C::BOX_BYTES), IDESC_O, (j | kk) ? 1u : 0u);
            umma_commit(&bar[PV_DONE + t]);
            umma_commit(&bar[V_EMPTY + t]);
            if (last) umma_commit(&bar[O_FULL + t]);
          }
        }
        ++nitem;
      }
      umma_commit(&bar[MMA_DONE]);  // TMEM stays allocated until every issued MMA is done
      mbar_wait(&bar[MMA_DONE], 0, err);
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ------------------------------------------------------------ softmax (row = TMEM lane)
    const int t = (warp - 4) >> 2;
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    const uint32_t tS = trow + t * BKV, tO = trow + C::T_O + t * DH;
    uint32_t g = 0, nitem = 0;
    bool ok = true;
    for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
      Item I;
      if (!item_at(it, cu, B, HP, n_tiles, Hq, Hkv, causal, I)) continue;
      const int qpos = I.q0 + r;  // query position in the sequence
      const int row_lim = qpos >= I.len ? 0 : (causal ? qpos + 1 : I.len);  // keys [0, row_lim) are visible
      float m = -INFINITY, l = 0.f;  // m: running max in log2 units
      for (int j = 0; j < I.nkv; ++j, ++g) {
        if (!mbar_wait_warp(&bar[S_FULL + t], g & 1, err)) { ok = false; break; }
        tc_fence_after();
        float v[BKV];
#pragma unroll
        for (int c = 0; c < BKV; c += 32) tmem_ld_32x32b_x32(tS + c, *reinterpret_cast<float(*)[32]>(v + c));
        tmem_ld_wait();
        const int lim = row_lim - j * BKV;
        if (lim < BKV) {
#pragma unroll
          for (int c = 0; c < BKV; ++c) v[c] = c < lim ? v[c] : -INFINITY;
        }
        float mx[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mx[e] = v[e];
#pragma unroll
        for (int c = 8; c < BKV; ++c) mx[c & 7] = fmaxf(mx[c & 7], v[c]);
        const float mb =
            fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])), fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7]))) *
            scale_log2;
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
        float pk[BKV / 2];  // bf16 pairs, bit-cast for tcgen05.st
#pragma unroll
        for (int e = 0; e < BKV / 2; ++e) {
          const float p0 = ex2(fmaf(v[2 * e], scale_log2, nm)), p1 = ex2(fmaf(v[2 * e + 1], scale_log2, nm));
          ls[(2 * e) & 7] += p0;
          ls[(2 * e + 1) & 7] += p1;
          pk[e] = __uint_as_float(pack_bf16x2(p0, p1));
        }
        l = l * corr + ((ls[0] + ls[1]) + (ls[2] + ls[3])) + ((ls[4] + ls[5]) + (ls[6] + ls[7]));
        if (__any_sync(0xffffffffu, moved)) {
          // O += P V of the previous block has finished with O (it completed
          // before this block's S was issued; the wait makes it explicit)
          if (!mbar_wait_warp(&bar[PV_DONE + t], (g - 1) & 1, err)) { ok = false; break; }
          tc_fence_after();
          float o[32];
#pragma unroll 1
          for (int c = 0; c < DH; c += 32) {
            tmem_ld_32x32b_x32(tO + c, o);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] *= corr;
            tmem_st_32x32b_x32(tO + c, o);
          }
        }
        tmem_st_32x32b_x32(tS, *reinterpret_cast<float(*)[32]>(pk));
        tmem_st_32x32b_x32(tS + 32, *reinterpret_cast<float(*)[32]>(pk + 32));
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar[P_FULL + t]);
      }
      if (!ok) break;
      // ---- O / l to global
      if (!mbar_wait_warp(&bar[O_FULL + t], nitem & 1, err)) { ok = false; break; }
      tc_fence_after();
      const float inv = l > 0.f ? 1.f / l : 0.f;
      const int h = t ? I.h1 : I.h0;
      const bool store = qpos < I.len && (t == 0 || I.h1 != I.h0);
      __nv_bfloat16* dst = out + (size_t)(I.s0 + qpos) * ld_out + h * DH;
      float o[32];
#pragma unroll 1
      for (int c = 0; c < DH; c += 32) {
        tmem_ld_32x32b_x32(tO + c, o);
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
      if (lane == 0) mbar_arrive(&bar[O_EMPTY + t]);
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
  CUtensorMap tm;
  if (!encode_tmap_2d(&tm, qkv, false, (uint64_t)rows_cap, (uint64_t)ld_qkv, 64, fa::BQ, nullptr))
    return cudaErrorInvalidValue;
  const int n_tiles = (max_len + fa::BQ - 1) / fa::BQ;
  const long n_items = (long)n_tiles * B * ((Hq + 1) / 2);
  const int grid = (int)std::min<long>(n_items, (long)device_sm_count());
  return launch_pdl(fa::attn_fa_kernel<DH>, dim3(grid), dim3(fa::NTHR), C::SMEM, st, tm,
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
