// Variable-length attention over packed sequences (cu_seqlens), causal for the
// LM prefill and bidirectional for the selector's cross-modal encoder (Eq. 3,
// Table 7(a)); grouped-query heads map query head i to kv head i / (Hq / Hkv).
// One tcgen05 kernel (below) serves both, head dims 64 and 128.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

// ===========================================================================
// tcgen05 flash attention.  One CTA = 128 query rows (TMEM lanes) of one head
// of one sequence, 6 warps, two CTAs per SM:
//   warp 0     TMA: the Q tile once, K and V tiles of 64 keys (two stages each)
//   warp 1     TMEM allocation; one thread issues S = Q K^T (M 128, N 64, both
//              K-major from shared memory) into one of two S buffers, and
//              O += P V with P read from Tensor Memory (where the softmax left
//              it, over its S buffer) and V an MN-major operand straight from
//              its TMA tile (no transpose); P is a bf16 hi + lo pair (two MMAs,
//              ~16 bits of P)
//   warps 2-5  softmax, one thread per query row: S row from TMEM, mask,
//              running max / sum in the exp2 domain, P back to TMEM, O
//              rescaled in TMEM only when the running max grows by more than
//              2^8 (P may then exceed 1 by up to 2^8: exact, since O and the
//              sum l share the stale max), final O / l to global
// TMEM columns: S / P buffers [0, 64) and [64, 128) (P: hi in the first 32
// columns, lo in the next 32, two bf16 per column), O [128, 128 + dh).
// Keys past the sequence get P = 0; their V rows must be finite (the caller
// keeps the rows past the packed length zero).
namespace tca {

constexpr int BQ = 128, BKV = 64, NTHR = 192;
constexpr float kRescaleLog2 = 8.f;  // rescale O once the max moved by more than this (log2 units)

template <int DH>
struct Cfg {
  static constexpr uint32_t Q_BYTES = BQ * DH * 2;    // DH/64 boxes of 128 rows x 128 B
  static constexpr uint32_t KV_BYTES = BKV * DH * 2;  // DH/64 boxes of 64 rows x 128 B
  static constexpr uint32_t OFF_Q = 0;
  static constexpr uint32_t OFF_K = OFF_Q + Q_BYTES;       // 2 stages
  static constexpr uint32_t OFF_V = OFF_K + 2 * KV_BYTES;  // 2 stages
  static constexpr uint32_t OFF_BAR = OFF_V + 2 * KV_BYTES;
  static constexpr size_t SMEM = 1024 + OFF_BAR + 128;
  static constexpr uint32_t TMEM_COLS = 256;
  static constexpr uint32_t T_O = 128;  // first O column
};

SP_DEVINL float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int DH>
__global__ void __launch_bounds__(NTHR, 2)
attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKV,
               __nv_bfloat16* __restrict__ out, const int* __restrict__ cu, int Hq, int Hkv, int ld_out,
               int causal, float scale_log2, int* err) {
  using C = Cfg<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = sm + C::OFF_Q;
  uint8_t* sK = sm + C::OFF_K;
  uint8_t* sV = sm + C::OFF_V;
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + C::OFF_BAR);
  uint64_t* q_full = bar + 0;
  uint64_t* k_full = bar + 1;     // [2] TMA
  uint64_t* k_empty = bar + 3;    // [2] S MMA commit
  uint64_t* v_full = bar + 5;     // [2] TMA
  uint64_t* v_empty = bar + 7;    // [2] P V MMA commit
  uint64_t* s_full = bar + 9;     // [2] S MMA commit
  uint64_t* s_empty = bar + 11;   // [2] P V MMA commit (the P that overlays S is consumed)
  uint64_t* p_full = bar + 13;    //     4 softmax warps
  uint64_t* o_done = bar + 14;    //     P V MMA commit
  uint64_t* mma_done = bar + 15;  //     every MMA of the CTA complete
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 16);

  pdl_wait();  // programmatic launch: the previous kernel's outputs are visible from here
  pdl_trigger();
  const int b = blockIdx.z, h = blockIdx.y;
  const int s0 = __ldg(cu + b);
  const int len = __ldg(cu + b + 1) - s0;
  // causal: the last query tiles see the most keys; launch them first
  const int q0 = (gridDim.x - 1 - blockIdx.x) * BQ;
  if (q0 >= len) return;
  const int kvh = h / (Hq / Hkv);
  const int qcol = h * DH, kcol = (Hq + kvh) * DH, vcol = (Hq + Hkv + kvh) * DH;
  const int kend = causal ? min(len, q0 + BQ) : len;
  const int n_kv = (kend + BKV - 1) / BKV;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
      mbar_init(&v_full[i], 1);
      mbar_init(&v_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&s_empty[i], 1);
    }
    mbar_init(p_full, 4);
    mbar_init(o_done, 1);
    mbar_init(mma_done, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tslot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmKV);
      mbar_arrive_expect_tx(q_full, C::Q_BYTES);
#pragma unroll
      for (int bx = 0; bx < DH / 64; ++bx) tma_load_2d(sQ + bx * (BQ * 128), &tmQ, q_full, qcol + bx * 64, s0 + q0);
      int issued = 0;
      for (int j = 0; j < n_kv; ++j) {
        const int st = j & 1;
        const uint32_t ph = ((j >> 1) & 1) ^ 1u;
        if (!mbar_wait(&k_empty[st], ph, err)) break;
        mbar_arrive_expect_tx(&k_full[st], C::KV_BYTES);
#pragma unroll
        for (int bx = 0; bx < DH / 64; ++bx)
          tma_load_2d(sK + st * C::KV_BYTES + bx * (BKV * 128), &tmKV, &k_full[st], kcol + bx * 64, s0 + j * BKV);
        if (!mbar_wait(&v_empty[st], ph, err)) break;
        mbar_arrive_expect_tx(&v_full[st], C::KV_BYTES);
#pragma unroll
        for (int bx = 0; bx < DH / 64; ++bx)
          tma_load_2d(sV + st * C::KV_BYTES + bx * (BKV * 128), &tmKV, &v_full[st], vcol + bx * 64, s0 + j * BKV);
        ++issued;
      }
      // the copies land before the CTA may exit (bounded waits)
      mbar_wait(q_full, 0, err);
      for (int j = max(0, issued - 2); j < issued; ++j) {
        mbar_wait(&k_full[j & 1], (j >> 1) & 1, err);
        mbar_wait(&v_full[j & 1], (j >> 1) & 1, err);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t IDESC_S = umma_idesc_bf16_f32(BQ, BKV);
      constexpr uint32_t IDESC_O = umma_idesc_bf16_f32(BQ, DH) | (1u << 16);  // B (V) MN-major
      bool ok = mbar_wait(q_full, 0, err);
      for (int j = 0; ok && j <= n_kv; ++j) {
        if (j < n_kv) {
          const int st = j & 1;
          const uint32_t ph = (j >> 1) & 1;
          if (!mbar_wait(&k_full[st], ph, err) || !mbar_wait(&s_empty[st], ph ^ 1u, err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sQ), b0 = smem_u32(sK + st * C::KV_BYTES);
#pragma unroll
          for (int kk = 0; kk < DH / 16; ++kk) {
            const uint32_t ao = (kk >> 2) * (BQ * 128) + (kk & 3) * 32;
            const uint32_t bo = (kk >> 2) * (BKV * 128) + (kk & 3) * 32;
            umma_bf16(tmem + st * BKV, umma_desc_sw128(a0 + ao), umma_desc_sw128(b0 + bo), IDESC_S, kk ? 1u : 0u);
          }
          umma_commit(&s_full[st]);
          umma_commit(&k_empty[st]);
        }
        if (j >= 1) {
          const int i = j - 1, st = i & 1;
          const uint32_t ph = (i >> 1) & 1;
          if (!mbar_wait(&v_full[st], ph, err) || !mbar_wait(p_full, i & 1, err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t bv = smem_u32(sV + st * C::KV_BYTES);
#pragma unroll
          for (int part = 0; part < 2; ++part) {
            const uint32_t ap = tmem + st * BKV + part * (BKV / 2);  // P hi / lo columns
#pragma unroll
            for (int kk = 0; kk < BKV / 16; ++kk)
              umma_bf16_ta(tmem + C::T_O, ap + kk * 8, umma_desc_sw128_mn(bv + kk * 2048, BKV * 128), IDESC_O,
                           (i | part | kk) ? 1u : 0u);
          }
          umma_commit(&v_empty[st]);
          umma_commit(&s_empty[st]);
          umma_commit(o_done);
        }
      }
      umma_commit(mma_done);  // TMEM stays allocated until every issued MMA is done
      mbar_wait(mma_done, 0, err);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax (row = TMEM lane)
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    const int qpos = q0 + r;  // query position in the sequence
    const int row_lim = qpos >= len ? 0 : (causal ? qpos + 1 : len);  // keys [0, row_lim) are visible
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    float m = -INFINITY, l = 0.f;  // m: running max in log2 units
    bool ok = true;
    for (int i = 0; ok && i < n_kv; ++i) {
      const int st = i & 1;
      if (!mbar_wait_warp(&s_full[st], (i >> 1) & 1, err)) { ok = false; break; }
      tc_fence_after();
      float v[BKV];
      tmem_ld_32x32b_x32(trow + st * BKV, *reinterpret_cast<float(*)[32]>(v));
      tmem_ld_32x32b_x32(trow + st * BKV + 32, *reinterpret_cast<float(*)[32]>(v + 32));
      tmem_ld_wait();
      const int lim = row_lim - i * BKV;
      float mx[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) mx[e] = -INFINITY;
#pragma unroll
      for (int c = 0; c < BKV; ++c) {
        v[c] = c < lim ? v[c] * scale_log2 : -INFINITY;
        mx[c & 7] = fmaxf(mx[c & 7], v[c]);
      }
      const float mb = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])), fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      // stale-max rule: move m (and rescale O and l) only when the block max exceeds it by > 2^8
      float corr = 1.f;
      bool moved = false;
      if (mb > m + kRescaleLog2 || (m == -INFINITY && mb > -INFINITY)) {
        corr = m == -INFINITY ? 0.f : ex2(m - mb);
        moved = m != -INFINITY;
        m = mb;
      }
      float ls[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) ls[e] = 0.f;
      const float mm = m == -INFINITY ? 0.f : m;
      float phi[BKV / 2], plo[BKV / 2];  // packed bf16 pairs, bit-cast for tcgen05.st
#pragma unroll
      for (int e = 0; e < BKV / 2; ++e) {
        const float p0 = ex2(v[2 * e] - mm), p1 = ex2(v[2 * e + 1] - mm);  // ex2(-inf) = 0
        ls[(2 * e) & 7] += p0;
        ls[(2 * e + 1) & 7] += p1;
        const uint32_t hw = pack_bf16x2(p0, p1);
        const float h0 = __uint_as_float(hw << 16), h1 = __uint_as_float(hw & 0xffff0000u);
        phi[e] = __uint_as_float(hw);
        plo[e] = __uint_as_float(pack_bf16x2(p0 - h0, p1 - h1));
      }
      l = l * corr + ((ls[0] + ls[1]) + (ls[2] + ls[3])) + ((ls[4] + ls[5]) + (ls[6] + ls[7]));
      if (i > 0) {
        // P V of the previous block has finished with O
        if (!mbar_wait_warp(o_done, (i - 1) & 1, err)) { ok = false; break; }
        tc_fence_after();
        if (__any_sync(0xffffffffu, moved)) {
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
      }
      tmem_st_32x32b_x32(trow + st * BKV, phi);
      tmem_st_32x32b_x32(trow + st * BKV + BKV / 2, plo);
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    // ---- O / l to global
    if (ok && mbar_wait_warp(o_done, (n_kv - 1) & 1, err)) {
      tc_fence_after();
      const float inv = l > 0.f ? 1.f / l : 0.f;
      __nv_bfloat16* dst = out + (size_t)(s0 + qpos) * ld_out + h * DH;
      float o[32];
#pragma unroll 1
      for (int c = 0; c < DH; c += 32) {
        tmem_ld_32x32b_x32(trow + C::T_O + c, o);
        tmem_ld_wait();
        if (qpos < len) {
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
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

}  // namespace tca
}  // namespace

template <int DH>
cudaError_t launch_attn_tc(const void* qkv, void* out, const int* cu, int B, int max_len, int rows_cap, int Hq,
                           int Hkv, bool causal, float scale_log2, int* err, cudaStream_t st) {
  using C = tca::Cfg<DH>;
  static bool attr = false;
  if (!attr) {
    cudaError_t r = cudaFuncSetAttribute(tca::attn_tc_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::SMEM);
    if (r != cudaSuccess) return r;
    attr = true;
  }
  const int ld_qkv = (Hq + 2 * Hkv) * DH;
  CUtensorMap tq, tkv;
  if (!encode_tmap_2d(&tq, qkv, false, (uint64_t)rows_cap, (uint64_t)ld_qkv, 64, tca::BQ, nullptr) ||
      !encode_tmap_2d(&tkv, qkv, false, (uint64_t)rows_cap, (uint64_t)ld_qkv, 64, tca::BKV, nullptr))
    return cudaErrorInvalidValue;
  dim3 grid((max_len + tca::BQ - 1) / tca::BQ, Hq, B);
  return launch_pdl(tca::attn_tc_kernel<DH>, grid, dim3(tca::NTHR), C::SMEM, st, tq, tkv,
                    reinterpret_cast<__nv_bfloat16*>(out), cu, Hq, Hkv, Hq * DH, causal ? 1 : 0, scale_log2, err);
}

cudaError_t attention_varlen(const void* qkv, void* out, const int* cu_seqlens, int B,
                             int max_seqlen_cap, int rows_cap, int Hq, int Hkv, int dh, bool causal,
                             int* err, cudaStream_t st) {
  if (B <= 0 || max_seqlen_cap <= 0 || rows_cap <= 0) return cudaSuccess;
  const float sl2 = 1.4426950408889634f / sqrtf((float)dh);
  prof_begin_launch(st);
  cudaError_t r = dh == 128 ? launch_attn_tc<128>(qkv, out, cu_seqlens, B, max_seqlen_cap, rows_cap, Hq, Hkv, causal,
                                                  sl2, err, st)
                : dh == 64  ? launch_attn_tc<64>(qkv, out, cu_seqlens, B, max_seqlen_cap, rows_cap, Hq, Hkv, causal,
                                                 sl2, err, st)
                            : cudaErrorInvalidValue;
  prof_end_launch(st, SP_K_ATTN, 0.0, 0.0);
  return r;
}

}  // namespace sp
