// Variable-length attention over packed sequences (cu_seqlens), causal for the
// LM prefill and bidirectional for the selector's cross-modal encoder (Eq. 3,
// Table 7(a)); grouped-query heads map query head i to kv head i / (Hq / Hkv).
// Two tcgen05 kernels (below), chosen by the longest sequence the call allows,
// serve both, head dims 64 and 128.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

// Sequences up to this many tokens take the head-pair kernel (two tiles in
// flight per CTA); longer ones the two-stream kernel with dynamic scheduling.
constexpr int kPairMaxLen = 1280;

// ===========================================================================
// Short sequences (up to kPairMaxLen keys): persistent tcgen05 flash attention
// over head pairs.  One CTA per SM walks a static list of work items (in chunks
// of sequences whose keys and values fit in L2, longest tiles first); an item
// is 128 query rows (one tile) of one sequence for a PAIR of query heads
// (2p, 2p + 1).  Two tiles (the pair's heads) are in flight per CTA, which is
// what keeps the tensor pipe busy when a tile has only one or two key blocks.
// Each head of the pair has its own pipeline in the CTA (its TMA thread, its
// two MMA-issuing threads, its softmax warpgroup, its TMEM columns); the two
// share the SM's tensor pipe, which interleaves them.
//
//   warps 0 / 3  TMA of head 0 / 1: the Q tile once per item, then per 64-key
//                block the K and V blocks into two-stage rings
//   warps 1 / 12 issue head 0 / 1's scores: S = Q K^T per 64-key block (M
//                128, N 64, both K-major from shared memory) into one of the
//                head's two S / P buffers (warp 1 also allocates the 512 TMEM
//                columns); S of block j + 2 reuses block j's buffer only once
//                O += P V of block j has completed (its commit)
//   warps 2 / 13 issue head 0 / 1's O += P V (P read from Tensor Memory where
//                the softmax wrote it over its S, V an MN-major operand straight
//                from its TMA block).  Two issuing threads per head let one's
//                barrier waits overlap the other's issue; two S / P buffers let
//                the softmax of block j overlap the scores of block j + 1.
//   warps 4-7   softmax of head 0, warps 8-11 of head 1: one thread per query
//               row (= TMEM lane): S row from TMEM, mask (causal diagonal
//               blocks, sequence tail), running max / sum in the exp2 domain, P
//               as bf16 back over S, O rescaled in TMEM only when the running
//               max grows by more than 2^8 (lazy rescale: O and the sum l share
//               the stale max, so the result is exact), final O / l to global.
// TMEM columns: S / P buffer b of head t at [128 t + 64 b, + 64) (P: 32
// columns of bf16 pairs over the first half of S), O of head t at
// [256 + DH t, + DH).
// Keys past the sequence get P = 0; their V rows must be finite (the caller
// keeps the rows past the packed length zero, or the tensor map ends there).
namespace fa_pair {

constexpr int BQ = 128, BKV = 64, NTHR = 448;
constexpr float kRescaleLog2 = 8.f;  // rescale O once the max moved by more than this (log2 units)

template <int DH>
struct Cfg {
  static constexpr uint32_t BOX_Q = BQ * 128;              // 128 rows x 64 bf16 (one 128-byte swizzle box)
  static constexpr uint32_t BOX_KV = BKV * 128;            // 64 rows x 64 bf16
  static constexpr uint32_t Q_BYTES = DH / 64 * BOX_Q;     // a Q tile of one head
  static constexpr uint32_t KV_BYTES = DH / 64 * BOX_KV;   // a K or V block of one head
  static constexpr uint32_t OFF_Q = 0;                     // [2 heads]
  static constexpr uint32_t OFF_K = 2 * Q_BYTES;           // [2 heads][2 stages]
  static constexpr uint32_t OFF_V = OFF_K + 4 * KV_BYTES;  // [2 heads][2 stages]
  static constexpr uint32_t OFF_BAR = OFF_V + 4 * KV_BYTES;
  static constexpr size_t SMEM_USED = 1024 + OFF_BAR + 512;
  // a CTA holds all 512 TMEM columns: ask for more than half of the shared
  // memory so that a second CTA is never co-resident (it would only wait)
  static constexpr size_t SMEM = SMEM_USED > 120 * 1024 ? SMEM_USED : 120 * 1024;
  static constexpr uint32_t T_O = 256;
};

// Barriers.  Per head t: Q_FULL + t, Q_EMPTY + t, O_FULL + t, O_EMPTY + t;
// per head t and stage / buffer b (= block index & 1): X + 2 t + b; per head t
// and issuer (0: scores, 1: P V): MMA_DONE + 2 t + issuer.
// A slot's K is free once the scores that read it are complete (S_FULL), its
// V once O += P V is (PV_DONE): no "empty" barriers.  The V block's bytes
// complete on the P-ready barrier of its block (four softmax warps plus the
// TMA thread's expect-tx arrive), so O += P V waits once for both.  Likewise
// the K barrier of block j counts two arrivals, the TMA's (with K's bytes) and
// the commit of O += P V of block j - 2 (the last reader of the S / P buffer
// block j's scores will overwrite; the TMA arrives twice for the first two
// blocks), so the scores wait once for both.
enum Bar {
  Q_FULL = 0, Q_EMPTY = 2, K_FULL = 4, S_FULL = 8, P_FULL = 12, PV_DONE = 16, O_FULL = 20, O_EMPTY = 22,
  MMA_DONE = 24, N_BARS = 28
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

struct Item {
  int s0, len, q0, h0, h1, kvh0, kvh1, nkv;
};

// Work item `it` of the static list.  The sequences go in chunks of S (sized
// on the host so that a chunk's keys and values stay in L2 while its items
// run); within a chunk, query tiles from the last (the most key blocks under a
// causal mask) to the first, then sequence, then head pair.  Returns false for
// tiles past the sequence's end.
SP_DEVINL bool item_at(int it, const int* __restrict__ cu, int B, int HP, int n_tiles, int S, int Hq, int Hkv,
                       bool causal, Item& I) {
  const int ch = it / (n_tiles * S * HP);
  const int b0 = ch * S, sc = min(S, B - b0);  // the chunk's first sequence and its sequence count
  const int rem0 = it - ch * (n_tiles * S * HP);
  const int per_tile = sc * HP;
  const int tile = n_tiles - 1 - rem0 / per_tile;
  const int rem = rem0 - (rem0 / per_tile) * per_tile;
  const int b = b0 + rem / HP, hp = rem - (rem / HP) * HP;
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
attn_pair_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKV,
               __nv_bfloat16* __restrict__ out, const int* __restrict__ cu, int B, int Hq, int Hkv, int n_tiles,
               int seq_chunk, int ld_out, int causal_i, float scale_log2, int* err) {
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
    for (int i = 0; i < N_BARS; ++i)
      mbar_init(&bar[i], (i >= P_FULL && i < P_FULL + 4) ? 5
                         : (i == O_EMPTY || i == O_EMPTY + 1) ? 4
                         : (i >= K_FULL && i < K_FULL + 4)    ? 2
                                                              : 1);
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

  if (warp == 0 || warp == 3) {
    // ------------------------------------------------------------ TMA of head t
    if (lane == 0) {
      const int t = warp == 3;
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmKV);
      uint32_t g = 0, nitem = 0;
      bool ok = true;
      uint8_t* sQ = sm + C::OFF_Q + t * C::Q_BYTES;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
        Item I;
        if (!item_at(it, cu, B, HP, n_tiles, seq_chunk, Hq, Hkv, causal, I)) continue;
        if (!mbar_wait(&bar[Q_EMPTY + t], (nitem & 1) ^ 1u, err)) break;
        mbar_arrive_expect_tx(&bar[Q_FULL + t], C::Q_BYTES);
        const int qcol = (t ? I.h1 : I.h0) * DH;
        const int kvh = t ? I.kvh1 : I.kvh0;
        const int kcol = (Hq + kvh) * DH, vcol = (Hq + Hkv + kvh) * DH;
#pragma unroll
        for (int bx = 0; bx < DH / 64; ++bx)
          tma_load_2d(sQ + bx * C::BOX_Q, &tmQ, &bar[Q_FULL + t], qcol + bx * 64, I.s0 + I.q0);
        for (int j = 0; j < I.nkv; ++j, ++g) {
          // slot st last held block g - 2: its K is free once that block's
          // scores are complete, its V once its O += P V is
          const uint32_t st = g & 1, pe = ((g >> 1) & 1) ^ 1u;
          uint8_t* sK = sm + C::OFF_K + (2 * t + st) * C::KV_BYTES;
          uint8_t* sV = sm + C::OFF_V + (2 * t + st) * C::KV_BYTES;
          uint64_t* kfull = &bar[K_FULL + 2 * t + st];
          uint64_t* vfull = &bar[P_FULL + 2 * t + st];
          if (g >= 2 && !mbar_wait(&bar[S_FULL + 2 * t + st], pe, err)) { ok = false; break; }
          mbar_arrive_expect_tx(kfull, C::KV_BYTES);
          if (g < 2) mbar_arrive(kfull);  // (no O += P V of block g - 2 arrives)
#pragma unroll
          for (int bx = 0; bx < DH / 64; ++bx)
            tma_load_2d(sK + bx * C::BOX_KV, &tmKV, kfull, kcol + bx * 64, I.s0 + j * BKV);
          if (g >= 2 && !mbar_wait(&bar[PV_DONE + 2 * t + st], pe, err)) { ok = false; ++g; break; }
          mbar_arrive_expect_tx(vfull, C::KV_BYTES);
#pragma unroll
          for (int bx = 0; bx < DH / 64; ++bx)
            tma_load_2d(sV + bx * C::BOX_KV, &tmKV, vfull, vcol + bx * 64, I.s0 + j * BKV);
        }
        ++nitem;
      }
      // every copy lands before the CTA may exit (bounded waits; normally
      // the consumers have waited for all of them already)
      if (nitem > 0) mbar_wait(&bar[Q_FULL + t], (nitem - 1) & 1, err);
      for (uint32_t gg = g >= 2 ? g - 2 : 0; gg < g; ++gg) {
        mbar_wait(&bar[K_FULL + 2 * t + (gg & 1)], (gg >> 1) & 1, err);
        mbar_wait(&bar[P_FULL + 2 * t + (gg & 1)], (gg >> 1) & 1, err);  // (V, and the block's P)
      }
    }
  } else if (warp == 1 || warp == 2 || warp >= 12) {
    // ------------------------------------------------------------ MMA issuers of head t
    // Two threads per head: one issues the scores, the other O += P V, so
    // that one's waits overlap the other's issue (tcgen05.commit tracks the
    // issuing thread's own MMAs, and the two never write the same columns).
    if (lane == 0) {
      const int t = warp >= 12 ? 1 : 0;
      const bool pv_issuer = warp == 2 || warp == 13;
      constexpr uint32_t IDESC_S = umma_idesc_bf16_f32(BQ, BKV);
      constexpr uint32_t IDESC_O = umma_idesc_bf16_f32(BQ, DH) | (1u << 16);  // B (V) MN-major
      // shared-memory descriptors of the stage bases; a K step adds its byte
      // offset / 16 to the address field (it stays below the field's 14 bits)
      const uint64_t dQ = umma_desc_sw128(smem_u32(sm + C::OFF_Q + t * C::Q_BYTES));
      const uint64_t dK0 = umma_desc_sw128(smem_u32(sm + C::OFF_K + 2 * t * C::KV_BYTES));
      const uint64_t dK1 = umma_desc_sw128(smem_u32(sm + C::OFF_K + (2 * t + 1) * C::KV_BYTES));
      const uint64_t dV0 = umma_desc_sw128_mn(smem_u32(sm + C::OFF_V + 2 * t * C::KV_BYTES), C::BOX_KV);
      const uint64_t dV1 = umma_desc_sw128_mn(smem_u32(sm + C::OFF_V + (2 * t + 1) * C::KV_BYTES), C::BOX_KV);
      const uint32_t tS = tmem + t * 128, tO = tmem + C::T_O + t * DH;
      uint32_t g = 0, nitem = 0;
      bool ok = true;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
        Item I;
        if (!item_at(it, cu, B, HP, n_tiles, seq_chunk, Hq, Hkv, causal, I)) continue;
        if (!pv_issuer) {
          // scores of every block: S(j) = Q K(j)^T into buffer j & 1
          ok = mbar_wait(&bar[Q_FULL + t], nitem & 1, err);
          for (int j = 0; ok && j < I.nkv; ++j) {
            const uint32_t gg = g + j, b = gg & 1, ph = (gg >> 1) & 1;
            // K_FULL also counts the completion of O += P V of block gg - 2,
            // the last reader of buffer b
            if (!mbar_wait(&bar[K_FULL + 2 * t + b], ph, err)) {
              ok = false;
              break;
            }
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < DH / 16; ++kk)
              umma_bf16(tS + b * BKV, dQ + (((kk >> 2) * C::BOX_Q + (kk & 3) * 32) >> 4),
                        (b ? dK1 : dK0) + (((kk >> 2) * C::BOX_KV + (kk & 3) * 32) >> 4), IDESC_S, kk ? 1u : 0u);
            umma_commit(&bar[S_FULL + 2 * t + b]);
            if (j + 1 == I.nkv) umma_commit(&bar[Q_EMPTY + t]);
          }
        } else {
          // O += P(j) V(j); P_FULL completes once the softmax wrote P and the
          // block's V landed
          for (int j = 0; ok && j < I.nkv; ++j) {
            const uint32_t gg = g + j, b = gg & 1, ph = (gg >> 1) & 1;
            if (!mbar_wait(&bar[P_FULL + 2 * t + b], ph, err) ||
                (j == 0 && !mbar_wait(&bar[O_EMPTY + t], (nitem & 1) ^ 1u, err))) {
              ok = false;
              break;
            }
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < BKV / 16; ++kk)
              umma_bf16_ta(tO, tS + b * BKV + kk * 8, (b ? dV1 : dV0) + ((kk * 2048) >> 4), IDESC_O,
                           (j | kk) ? 1u : 0u);
            umma_commit(&bar[PV_DONE + 2 * t + b]);
            umma_commit(&bar[K_FULL + 2 * t + b]);  // (counts toward block gg + 2's K barrier)
            if (j + 1 == I.nkv) umma_commit(&bar[O_FULL + t]);
          }
        }
        g += I.nkv;
        ++nitem;
      }
      // TMEM stays allocated until every MMA this thread issued is done
      umma_commit(&bar[MMA_DONE + 2 * t + (pv_issuer ? 1 : 0)]);
      mbar_wait(&bar[MMA_DONE + 2 * t + (pv_issuer ? 1 : 0)], 0, err);
    }
    __syncwarp();
  } else if (warp >= 4 && warp < 12) {
    // ------------------------------------------------------------ softmax (row = TMEM lane)
    const int t = (warp - 4) >> 2;
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    const uint32_t tS = trow + t * 128, tO = trow + C::T_O + t * DH;
    uint32_t g = 0, nitem = 0;
    bool ok = true;
    for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
      Item I;
      if (!item_at(it, cu, B, HP, n_tiles, seq_chunk, Hq, Hkv, causal, I)) continue;
      const int qpos = I.q0 + r;  // query position in the sequence
      const int row_lim = qpos >= I.len ? 0 : (causal ? qpos + 1 : I.len);  // keys [0, row_lim) are visible
      float m = -INFINITY, l = 0.f;  // m: running max in log2 units
      for (int j = 0; j < I.nkv; ++j, ++g) {
        const uint32_t b = g & 1;
        if (!mbar_wait_warp(&bar[S_FULL + 2 * t + b], (g >> 1) & 1, err)) { ok = false; break; }
        tc_fence_after();
        float v[BKV];
        tmem_ld_32x32b_x32(tS + b * BKV, *reinterpret_cast<float(*)[32]>(v));
        tmem_ld_32x32b_x32(tS + b * BKV + 32, *reinterpret_cast<float(*)[32]>(v + 32));
        tmem_ld_wait();
        const int lim = row_lim - j * BKV;
        if (lim < BKV) {
#pragma unroll
          for (int c = 0; c < BKV; ++c) v[c] = c < lim ? v[c] : -INFINITY;
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
        const float mb = max3(max3(mx[0], mx[1], mx[2]), max3(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7])) * scale_log2;
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
          // O += P V of the previous block must be done with O before it is rescaled
          if (!mbar_wait_warp(&bar[PV_DONE + 2 * t + ((g - 1) & 1)], ((g - 1) >> 1) & 1, err)) { ok = false; break; }
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
        tmem_st_32x32b_x32(tS + b * BKV, pk);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar[P_FULL + 2 * t + b]);
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

}  // namespace fa_pair

// ===========================================================================
// Longer sequences: persistent tcgen05 flash attention.  One CTA per SM takes
// work items from a global ticket counter (the last CTA out leaves it zero for
// the next launch; without a counter, a static stride); an item is 128 query
// rows (one tile) of one head of one sequence.  Within chunks of sequences whose
// keys and values fit in L2, the item list runs from the tiles with the most
// key blocks to those with the fewest, so that the dynamic assignment balances
// the SMs.
//
//   warp 0      scheduler + TMA: takes the tickets, publishes each item to the
//               other roles through a four-entry ring in shared memory, and loads
//               the Q tile once per item, then per 128-key block the K block into
//               a three-slot ring
//   warp 3      TMA of the V blocks into a two-slot ring (a thread of its own, so
//               that waiting for a free V slot never holds back the next K)
//   warp 1      issues the scores S = Q K^T (M 128, N 128, both K-major from
//               shared memory) into one of three S / P buffers in TMEM; it also
//               allocates the 512 TMEM columns
//   warp 2      issues O += P V (P read from Tensor Memory where the softmax
//               wrote it over its S, V an MN-major operand straight from its
//               TMA block)
//   warps 4-7   softmax stream 0: the even key blocks (counted over the CTA's
//   warps 8-11  whole walk); stream 1: the odd blocks.  A thread owns one query
//               row (= TMEM lane) of its stream's blocks, all 128 columns.
// The two streams work on consecutive blocks at the same time and share one O
// accumulator, so both must scale a block's P by the same running max m.  m
// changes only when a block's max exceeds it by more than 2^8 (lazy rescale:
// P <= 2^8, and O and the sums are rescaled on a change, so the result is
// exact); each block publishes its m for the next one through shared memory
// (an mbarrier per parity of the block, bounded waits).  Waiting for the
// previous block's m costs a row max, not a softmax: the exponentials of the
// two streams overlap.  Each stream keeps its own partial row sum with its own
// reference max; at the end of an item both are brought to the last m and
// added.  A block that moves m rescales O in TMEM once O += P V of the block
// before has completed.  The final O / l goes to global memory, each stream
// storing half of the head dims: a warp releases O as soon as it has read its
// columns, then stores its 32 rows through a small shared-memory stage so that
// every store instruction writes whole 64-byte row segments.
// Three S / P buffers let the scores run up to two blocks ahead; the scores of
// block j + 3 reuse block j's buffer only once O += P V of block j has
// completed.  Each issuing thread waits once per block: the K barrier of block
// j counts the TMA's arrival (with K's bytes) and the commit of O += P V of
// block j - 3; the P barrier counts the stream's four softmax warps and the
// TMA's arrival with V's bytes.  A K slot is free once the scores that read it
// are complete, a V slot once O += P V is: no "empty" barriers.
// TMEM columns: S / P buffer b at [128 b, 128 b + 128) (P: 64 columns of bf16
// pairs over the first half of S), O at [384, 384 + DH).
// Keys past the sequence get P = 0; their V rows must be finite (the caller
// keeps the rows past the packed length zero, or the tensor map ends there).
namespace fa {

constexpr int BQ = 128, BKV = 128, NTHR = 384, NSB = 3, NVS = 2, NIR = 4;
constexpr float kRescaleLog2 = 8.f;  // rescale O once the max moved by more than this (log2 units)

// Barriers; X + s for the slot / buffer s of a block, M_FULL + (block & 1) for
// the running-max hand-off, IT_FULL / IT_EMPTY + entry of the item ring.
enum Bar {
  Q_FULL = 0, Q_EMPTY = 1, K_FULL = 2, S_FULL = 5, P_FULL = 8, PV_DONE = 11, O_FULL = 14, O_EMPTY = 15,
  MMA_DONE = 16, M_FULL = 18, XL = 20, IT_FULL = 21, IT_EMPTY = 25, N_BARS = 29
};

template <int DH>
struct Cfg {
  static constexpr uint32_t BOX = 128 * 128;               // 128 rows x 64 bf16 (one 128-byte swizzle box)
  static constexpr uint32_t TILE = DH / 64 * BOX;          // a Q tile or a K / V block
  static constexpr uint32_t OFF_Q = 0;
  static constexpr uint32_t OFF_K = TILE;                  // [NSB]
  static constexpr uint32_t OFF_V = OFF_K + NSB * TILE;    // [NVS]
  static constexpr uint32_t OFF_M = OFF_V + NVS * TILE;    // running max per block parity: [2][128] floats
  static constexpr uint32_t OFF_L = OFF_M + 2 * 128 * 4;   // row sums: [item parity][stream][128] floats
  static constexpr uint32_t OFF_RING = OFF_L + 4 * 128 * 4;  // item ring: [NIR][8] ints
  static constexpr uint32_t OFF_STG = OFF_RING + NIR * 32;   // output stage: [8 warps][32 rows][64 B]
  static constexpr uint32_t OFF_BAR = OFF_STG + 8 * 2048;
  static constexpr size_t SMEM_USED = 1024 + OFF_BAR + N_BARS * 8 + 16;
  // a CTA holds all 512 TMEM columns: ask for more than half of the shared
  // memory so that a second CTA is never co-resident (it would only wait)
  static constexpr size_t SMEM = SMEM_USED > 120 * 1024 ? SMEM_USED : 120 * 1024;
  static constexpr uint32_t T_O = 384;
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

struct Item {
  int s0, len, q0, h, kvh, nkv;  // nkv == 0: no more items
};

// Work item `it` of the list.  The sequences go in chunks of S (sized on the
// host so that a chunk's keys and values stay in L2 while its items run);
// within a chunk, query tiles from the last (the most key blocks under a causal
// mask) to the first, then sequence, then head.  Returns false for tiles past
// the sequence's end.
SP_DEVINL bool item_at(int it, const int* __restrict__ cu, int B, int Hq, int n_tiles, int S, int Hkv, bool causal,
                       Item& I) {
  const int ch = it / (n_tiles * S * Hq);
  const int b0 = ch * S, sc = min(S, B - b0);  // the chunk's first sequence and its sequence count
  const int rem0 = it - ch * (n_tiles * S * Hq);
  const int per_tile = sc * Hq;
  const int tile = n_tiles - 1 - rem0 / per_tile;
  const int rem = rem0 - (rem0 / per_tile) * per_tile;
  const int b = b0 + rem / Hq;
  I.h = rem - (rem / Hq) * Hq;
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
               int seq_chunk, int ld_out, int causal_i, float scale_log2, int* sched, int* err) {
  using C = Cfg<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + C::OFF_BAR);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + N_BARS);
  float* mchain = reinterpret_cast<float*>(sm + C::OFF_M);
  float* lsum = reinterpret_cast<float*>(sm + C::OFF_L);
  int* ring = reinterpret_cast<int*>(sm + C::OFF_RING);
  const bool causal = causal_i != 0;
  const int n_items = n_tiles * B * Hq;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < N_BARS; ++i) {
      uint32_t n = 1;
      if (i >= K_FULL && i < K_FULL + NSB) n = 2;   // TMA + O += P V of block - 3
      if (i >= P_FULL && i < P_FULL + NSB) n = 5;   // the stream's 4 softmax warps + TMA (V)
      if (i == O_EMPTY || i == XL) n = 8;           // all softmax warps
      if (i == M_FULL || i == M_FULL + 1) n = 4;    // the publishing stream's warps
      if (i >= IT_EMPTY) n = 11;                    // both issuers, the V loader, 8 softmax warps
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

  // consumers' view of the item ring: entry ri % NIR, phase ri / NIR
  auto take_item = [&](uint32_t ri, Item& I) -> bool {
    const uint32_t e = ri % NIR;
    if (!mbar_wait_warp(&bar[IT_FULL + e], (ri / NIR) & 1, err)) return false;
    const int* r = ring + e * 8;
    I.s0 = r[0]; I.len = r[1]; I.q0 = r[2]; I.h = r[3]; I.kvh = r[4]; I.nkv = r[5];
    __syncwarp();
    if (lane == 0) mbar_arrive(&bar[IT_EMPTY + e]);
    return true;
  };

  if (warp == 0) {
    // ------------------------------------------------------------ scheduler + TMA
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmKV);
      int k = 0;
      auto fetch = [&]() -> int {
        ++k;
        return sched ? (int)gridDim.x + atomicAdd(sched, 1) : (int)blockIdx.x + k * (int)gridDim.x;
      };
      int ticket = blockIdx.x;
      int nxt = ticket < n_items ? fetch() : n_items;  // one ticket ahead: the atomic's latency overlaps
      uint32_t g = 0, ni = 0;
      bool ok = true;
      while (ok) {
        Item I;
        bool have = false;
        while (!have && ticket < n_items) {
          have = item_at(ticket, cu, B, Hq, n_tiles, seq_chunk, Hkv, causal, I);
          ticket = nxt;
          nxt = ticket < n_items ? fetch() : n_items;
        }
        const uint32_t e = ni % NIR;
        if (ni >= NIR && !mbar_wait(&bar[IT_EMPTY + e], ((ni / NIR) & 1) ^ 1u, err)) break;
        int* r = ring + e * 8;
        if (have) {
          r[0] = I.s0; r[1] = I.len; r[2] = I.q0; r[3] = I.h; r[4] = I.kvh; r[5] = I.nkv;
        } else {
          r[5] = 0;
        }
        mbar_arrive(&bar[IT_FULL + e]);
        if (!have) break;
        if (!mbar_wait(&bar[Q_EMPTY], (ni & 1) ^ 1u, err)) break;
        ++ni;
        mbar_arrive_expect_tx(&bar[Q_FULL], C::TILE);
#pragma unroll
        for (int bx = 0; bx < DH / 64; ++bx)
          tma_load_2d(sm + C::OFF_Q + bx * C::BOX, &tmQ, &bar[Q_FULL], I.h * DH + bx * 64, I.s0 + I.q0);
        const int kcol = (Hq + I.kvh) * DH;
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
        }
      }
      // every copy lands before the CTA may exit (bounded waits; normally
      // the consumers have waited for all of them already)
      if (ni > 0) mbar_wait(&bar[Q_FULL], (ni - 1) & 1, err);
      for (uint32_t gg = g >= NSB ? g - NSB : 0; gg < g; ++gg) mbar_wait(&bar[K_FULL + gg % NSB], (gg / NSB) & 1, err);
    }
  } else if (warp == 3) {
    // ------------------------------------------------------------ TMA of V
    uint32_t g = 0, ri = 0;
    bool ok = true;
    while (ok) {
      Item I;
      if (!take_item(ri++, I) || I.nkv == 0) break;
      if (lane == 0) {
        const int vcol = (Hq + Hkv + I.kvh) * DH;
        for (int j = 0; j < I.nkv; ++j) {
          const uint32_t gg = g + j;
          // V slot gg % 2 last held block gg - 2: free once its O += P V is complete
          if (gg >= NVS && !mbar_wait(&bar[PV_DONE + (gg - NVS) % NSB], ((gg - NVS) / NSB) & 1, err)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&bar[P_FULL + gg % NSB], C::TILE);
#pragma unroll
          for (int bx = 0; bx < DH / 64; ++bx)
            tma_load_2d(sm + C::OFF_V + (gg % NVS) * C::TILE + bx * C::BOX, &tmKV, &bar[P_FULL + gg % NSB],
                        vcol + bx * 64, I.s0 + j * BKV);
        }
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      g += I.nkv;
    }
    if (lane == 0)  // the last copies land before the CTA may exit (the block's P completes the same barrier)
      for (uint32_t gg = g >= NSB ? g - NSB : 0; gg < g; ++gg) mbar_wait(&bar[P_FULL + gg % NSB], (gg / NSB) & 1, err);
    __syncwarp();
  } else if (warp == 1 || warp == 2) {
    // ------------------------------------------------------------ MMA issuers
    // warp 1: the scores; warp 2: O += P V (tcgen05.commit tracks the issuing
    // thread's own MMAs; the two write disjoint TMEM columns)
    const bool pv_issuer = warp == 2;
    constexpr uint32_t IDESC_S = umma_idesc_bf16_f32(BQ, BKV);
    constexpr uint32_t IDESC_O = umma_idesc_bf16_f32(BQ, DH) | (1u << 16);  // B (V) MN-major
    // shared-memory descriptors of the slot bases; a K step adds its byte
    // offset / 16 to the address field (it stays below the field's 14 bits)
    const uint64_t dQ = umma_desc_sw128(smem_u32(sm + C::OFF_Q));
    const uint64_t dK = umma_desc_sw128(smem_u32(sm + C::OFF_K));
    const uint64_t dV = umma_desc_sw128_mn(smem_u32(sm + C::OFF_V), C::BOX);
    const uint64_t slot16 = C::TILE >> 4;
    uint32_t g = 0, nitem = 0, ri = 0;
    bool ok = true;
    while (ok) {
      Item I;
      if (!take_item(ri++, I) || I.nkv == 0) break;
      if (lane == 0) {
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
            // P_FULL completes once the stream's softmax wrote P and the block's V landed
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
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      g += I.nkv;
      ++nitem;
    }
    if (lane == 0) {
      // TMEM stays allocated until every MMA this thread issued is done
      umma_commit(&bar[MMA_DONE + (pv_issuer ? 1 : 0)]);
      mbar_wait(&bar[MMA_DONE + (pv_issuer ? 1 : 0)], 0, err);
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ------------------------------------------------------------ softmax streams (row = TMEM lane)
    const uint32_t s = (uint32_t)(warp - 4) >> 2;
    const int r = (warp & 3) * 32 + lane;
    const uint32_t trow = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    uint32_t g = 0, nitem = 0, ri = 0;
    bool ok = true;
    while (ok) {
      Item I;
      if (!take_item(ri++, I) || I.nkv == 0) break;
      const int qpos = I.q0 + r;  // query position in the sequence
      const int row_lim = qpos >= I.len ? 0 : (causal ? qpos + 1 : I.len);  // keys [0, row_lim) are visible
      float mlast = -INFINITY;  // m of this stream's latest block
      float ms = -INFINITY, ls = 0.f;  // this stream's partial row sum, relative to 2^ms
      for (int j = (int)((g & 1) != s); j < I.nkv; j += 2) {
        const uint32_t gg = g + j, sb = gg % NSB;
        if (!mbar_wait_warp(&bar[S_FULL + sb], (gg / NSB) & 1, err)) { ok = false; break; }
        tc_fence_after();
        float v[BKV];
#pragma unroll
        for (int c = 0; c < BKV / 32; ++c)
          tmem_ld_32x32b_x32(trow + sb * BKV + c * 32, *reinterpret_cast<float(*)[32]>(v + c * 32));
        tmem_ld_wait();
        const int lim = row_lim - j * BKV;
        if (lim < BKV) {
#pragma unroll
          for (int c = 0; c < BKV; ++c) v[c] = c < lim ? v[c] : -INFINITY;
        }
        float mx[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mx[e] = max3(v[e], v[e + 8], v[e + 16]);
#pragma unroll
        for (int c = 24; c + 16 <= BKV; c += 16) {
#pragma unroll
          for (int e = 0; e < 8; ++e) mx[e] = max3(mx[e], v[c + e], v[c + 8 + e]);
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) mx[e] = fmaxf(mx[e], v[BKV - 8 + e]);
        const float mh = max3(max3(mx[0], mx[1], mx[2]), max3(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7]));
        // m of the previous block of this item (the other stream's), then this block's
        float mp = -INFINITY;
        if (j > 0) {
          const uint32_t pb = gg - 1;
          if (!mbar_wait_warp(&bar[M_FULL + (pb & 1)], (pb >> 1) & 1, err)) { ok = false; break; }
          mp = mchain[(pb & 1) * 128 + r];
        }
        const float mb = mh * scale_log2;
        float m = mp, corr = 1.f;
        bool moved = false;
        if (mb > mp + kRescaleLog2 || (mp == -INFINITY && mb > -INFINITY)) {
          corr = mp == -INFINITY ? 0.f : ex2(mp - mb);
          moved = mp != -INFINITY;
          m = mb;
        }
        mchain[(gg & 1) * 128 + r] = m;
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar[M_FULL + (gg & 1)]);
        mlast = m;
        if (m != ms) {  // bring this stream's partial sum to the new reference
          ls = ms == -INFINITY ? 0.f : ls * ex2(ms - m);
          ms = m;
        }
        const float nm = m == -INFINITY ? 0.f : -m;
        float rs[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) rs[e] = 0.f;
#pragma unroll
        for (int c = 0; c < BKV / 32; ++c) {
          float pk[16];  // bf16 pairs, bit-cast for tcgen05.st
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const float p0 = ex2(fmaf(v[c * 32 + 2 * e], scale_log2, nm));
            const float p1 = ex2(fmaf(v[c * 32 + 2 * e + 1], scale_log2, nm));
            rs[(2 * e) & 7] += p0;
            rs[(2 * e + 1) & 7] += p1;
            pk[e] = __uint_as_float(pack_bf16x2(p0, p1));
          }
          tmem_st_cols<16>(trow + sb * BKV + c * 16, pk);
        }
        ls += ((rs[0] + rs[1]) + (rs[2] + rs[3])) + ((rs[4] + rs[5]) + (rs[6] + rs[7]));
        if (__any_sync(0xffffffffu, moved)) {
          // O += P V of the previous block must be done with O before it is rescaled
          const uint32_t pb = gg - 1;
          if (!mbar_wait_warp(&bar[PV_DONE + pb % NSB], (pb / NSB) & 1, err)) { ok = false; break; }
          tc_fence_after();
          float o[32];
#pragma unroll 1
          for (int c = 0; c < DH; c += 32) {
            tmem_ld_32x32b_x32(trow + C::T_O + c, o);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] *= corr;
            tmem_st_32x32b_x32(trow + C::T_O + c, o);
          }
        }
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar[P_FULL + sb]);
      }
      if (!ok) break;
      // ---- O / l to global: l is the two streams' partial sums at the last block's m
      const uint32_t last = g + I.nkv - 1;
      if ((last & 1) != s) {
        if (!mbar_wait_warp(&bar[M_FULL + (last & 1)], (last >> 1) & 1, err)) { ok = false; break; }
        mlast = mchain[(last & 1) * 128 + r];
      }
      const float lsc = (ms == -INFINITY || mlast == -INFINITY) ? 0.f : ls * ex2(ms - mlast);
      float* xl = lsum + (nitem & 1) * 256;
      xl[s * 128 + r] = lsc;
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar[XL]);
      if (!mbar_wait_warp(&bar[XL], nitem & 1, err)) { ok = false; break; }
      const float lt = xl[r] + xl[128 + r];
      if (!mbar_wait_warp(&bar[O_FULL], nitem & 1, err)) { ok = false; break; }
      tc_fence_after();
      constexpr int HD = DH / 2;  // this stream's head dims
      float o[HD];
#pragma unroll
      for (int c = 0; c < HD; c += 32)
        tmem_ld_32x32b_x32(trow + C::T_O + s * HD + c, *reinterpret_cast<float(*)[32]>(o + c));
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar[O_EMPTY]);  // O may be overwritten from here
      const float inv = lt > 0.f ? 1.f / lt : 0.f;
      // stage: row `lane` of this warp, 32 columns (64 bytes) per pass; 16-byte
      // granule q of a row sits at q ^ ((row >> 1) & 3) (no bank conflicts)
      uint8_t* stg = sm + C::OFF_STG + (warp - 4) * 2048;
      const int rows_left = I.len - (I.q0 + (warp & 3) * 32);  // valid rows of this warp's 32
      __nv_bfloat16* dst0 = out + (size_t)(I.s0 + I.q0 + (warp & 3) * 32) * ld_out + I.h * DH + s * HD;
#pragma unroll
      for (int c = 0; c < HD; c += 32) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint4 u;
          u.x = pack_bf16x2(o[c + 8 * q + 0] * inv, o[c + 8 * q + 1] * inv);
          u.y = pack_bf16x2(o[c + 8 * q + 2] * inv, o[c + 8 * q + 3] * inv);
          u.z = pack_bf16x2(o[c + 8 * q + 4] * inv, o[c + 8 * q + 5] * inv);
          u.w = pack_bf16x2(o[c + 8 * q + 6] * inv, o[c + 8 * q + 7] * inv);
          *reinterpret_cast<uint4*>(stg + lane * 64 + ((q ^ ((lane >> 1) & 3)) * 16)) = u;
        }
        __syncwarp();
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int row = k * 8 + (lane >> 2), q = lane & 3;
          const uint4 u = *reinterpret_cast<const uint4*>(stg + row * 64 + ((q ^ ((row >> 1) & 3)) * 16));
          if (row < rows_left) *reinterpret_cast<uint4*>(dst0 + (size_t)row * ld_out + c + q * 8) = u;
        }
        __syncwarp();
      }
      g += I.nkv;
      ++nitem;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
  // the last CTA out leaves the ticket counter zero for the next launch
  if (threadIdx.x == 0 && sched) {
    __threadfence();
    if (atomicAdd(sched + 1, 1) == (int)gridDim.x - 1) {
      atomicExch(sched, 0);
      atomicExch(sched + 1, 0);
    }
  }
}

}  // namespace fa
}  // namespace

// Sequences per item chunk: as many as keep their keys and values (at the
// longest length the call allows) within 48 MB of the L2, at least one.
static int attn_seq_chunk(int max_len, int Hkv, int dh, int B) {
  const double kv = (double)max_len * Hkv * dh * 2 * 2;
  const int s = kv > 0 ? (int)(48e6 / kv) : B;
  return std::max(1, std::min(s, B));
}

template <int DH>
cudaError_t launch_attn_fa(const void* qkv, void* out, const int* cu, int B, int max_len, int rows_cap, int Hq,
                           int Hkv, bool causal, float scale_log2, int* sched, int* err, cudaStream_t st) {
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
  const int seq_chunk = attn_seq_chunk(max_len, Hkv, DH, B);
  const long n_items = (long)n_tiles * B * Hq;
  const int grid = (int)std::min<long>(n_items, (long)device_sm_count());
  return launch_pdl(fa::attn_fa_kernel<DH>, dim3(grid), dim3(fa::NTHR), C::SMEM, st, tq, tkv,
                    reinterpret_cast<__nv_bfloat16*>(out), cu, B, Hq, Hkv, n_tiles, seq_chunk, Hq * DH,
                    causal ? 1 : 0,
                    scale_log2, sched, err);
}

template <int DH>
cudaError_t launch_attn_pair(const void* qkv, void* out, const int* cu, int B, int max_len, int rows_cap, int Hq,
                           int Hkv, bool causal, float scale_log2, int* err, cudaStream_t st) {
  using C = fa_pair::Cfg<DH>;
  static bool attr = false;
  if (!attr) {
    cudaError_t r = cudaFuncSetAttribute(fa_pair::attn_pair_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::SMEM);
    if (r != cudaSuccess) return r;
    attr = true;
  }
  if (Hkv <= 0 || Hq % Hkv != 0) return cudaErrorInvalidValue;
  const int ld_qkv = (Hq + 2 * Hkv) * DH;
  CUtensorMap tq, tkv;
  if (!encode_tmap_2d(&tq, qkv, false, (uint64_t)rows_cap, (uint64_t)ld_qkv, 64, fa_pair::BQ, nullptr) ||
      !encode_tmap_2d(&tkv, qkv, false, (uint64_t)rows_cap, (uint64_t)ld_qkv, 64, fa_pair::BKV, nullptr))
    return cudaErrorInvalidValue;
  const int n_tiles = (max_len + fa_pair::BQ - 1) / fa_pair::BQ;
  const int seq_chunk = attn_seq_chunk(max_len, Hkv, DH, B);
  const long n_items = (long)n_tiles * B * ((Hq + 1) / 2);
  const int grid = (int)std::min<long>(n_items, (long)device_sm_count());
  return launch_pdl(fa_pair::attn_pair_kernel<DH>, dim3(grid), dim3(fa_pair::NTHR), C::SMEM, st, tq, tkv,
                    reinterpret_cast<__nv_bfloat16*>(out), cu, B, Hq, Hkv, n_tiles, seq_chunk, Hq * DH,
                    causal ? 1 : 0,
                    scale_log2, err);
}

cudaError_t attention_varlen(const void* qkv, void* out, const int* cu_seqlens, int B,
                             int max_seqlen_cap, int rows_cap, int Hq, int Hkv, int dh, bool causal,
                             int* sched, int* err, cudaStream_t st) {
  if (B <= 0 || max_seqlen_cap <= 0 || rows_cap <= 0) return cudaSuccess;
  const float sl2 = 1.4426950408889634f / sqrtf((float)dh);
  prof_begin_launch(st);
  const bool pair = max_seqlen_cap <= kPairMaxLen;
  cudaError_t r = cudaErrorInvalidValue;
  if (dh == 128)
    r = pair ? launch_attn_pair<128>(qkv, out, cu_seqlens, B, max_seqlen_cap, rows_cap, Hq, Hkv, causal, sl2, err, st)
             : launch_attn_fa<128>(qkv, out, cu_seqlens, B, max_seqlen_cap, rows_cap, Hq, Hkv, causal, sl2, sched,
                                   err, st);
  else if (dh == 64)
    r = pair ? launch_attn_pair<64>(qkv, out, cu_seqlens, B, max_seqlen_cap, rows_cap, Hq, Hkv, causal, sl2, err, st)
             : launch_attn_fa<64>(qkv, out, cu_seqlens, B, max_seqlen_cap, rows_cap, Hq, Hkv, causal, sl2, sched,
                                  err, st);
  prof_end_launch(st, SP_K_ATTN, 0.0, 0.0);
  return r;
}

}  // namespace sp
