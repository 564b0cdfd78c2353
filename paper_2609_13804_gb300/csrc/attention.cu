// Variable-length attention over packed sequences (cu_seqlens), causal for the
// LM prefill and bidirectional for the selector's cross-modal encoder (Eq. 3,
// Table 7(a)); grouped-query heads map query head i to kv head i / (Hq / Hkv).
//
// One CTA = 64 query rows of one head of one sequence (4 warps x 16 rows).
// K/V tiles of 64 keys are double-buffered in shared memory with cp.async
// (16-byte chunks, XOR-swizzled per row), S = Q K^T and O += P V use bf16
// mma.sync with fp32 accumulators and an online softmax in the exp2 domain.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

constexpr int BQ = 64, BKV = 64;

SP_DEVINL uint32_t swz(int r, int c, int dh) {  // element offset of (row, col), col % 8 == 0
  return (uint32_t)(r * dh + ((((c >> 3) ^ (r & 7))) << 3));
}

SP_DEVINL void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int sz = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(sz) : "memory");
}
SP_DEVINL void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
SP_DEVINL void cp_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

SP_DEVINL void ldsm_x4(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c, uint32_t& d) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(a), "=r"(b), "=r"(c), "=r"(d) : "r"(addr));
}
SP_DEVINL void ldsm_x4_t(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c, uint32_t& d) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(a), "=r"(b), "=r"(c), "=r"(d) : "r"(addr));
}
SP_DEVINL void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <int DH>
__global__ void __launch_bounds__(128)
attn_kernel(const __nv_bfloat16* __restrict__ qkv, __nv_bfloat16* __restrict__ out,
            const int* __restrict__ cu, int Hq, int Hkv, int ld_qkv, int ld_out, int causal,
            float scale_log2) {
  extern __shared__ __align__(128) __nv_bfloat16 sm[];
  __nv_bfloat16* Qs = sm;
  __nv_bfloat16* Ks = sm + BQ * DH;
  __nv_bfloat16* Vs = Ks + 2 * BKV * DH;

  const int b = blockIdx.z, h = blockIdx.y;
  const int s0 = __ldg(cu + b);
  const int len = __ldg(cu + b + 1) - s0;
  const int q0 = blockIdx.x * BQ;
  if (q0 >= len) return;
  const int kvh = h / (Hq / Hkv);
  const int qcol = h * DH, kcol = (Hq + kvh) * DH, vcol = (Hq + Hkv + kvh) * DH;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr int CH = DH / 8;  // 16-byte chunks per row

  // Q tile
  for (int i = tid; i < BQ * CH; i += 128) {
    const int r = i / CH, c = (i % CH) * 8;
    const bool ok = q0 + r < len;
    const __nv_bfloat16* src = qkv + (size_t)(s0 + (ok ? q0 + r : 0)) * ld_qkv + qcol + c;
    cp_async16(smem_u32(Qs + swz(r, c, DH)), src, ok);
  }
  const int kend = causal ? min(len, q0 + BQ) : len;
  const int n_kt = (kend + BKV - 1) / BKV;
  auto load_kv = [&](int kt, int buf) {
    __nv_bfloat16* kd = Ks + buf * BKV * DH;
    __nv_bfloat16* vd = Vs + buf * BKV * DH;
    for (int i = tid; i < BKV * CH; i += 128) {
      const int r = i / CH, c = (i % CH) * 8;
      const int key = kt * BKV + r;
      const bool ok = key < len;
      const size_t row = (size_t)(s0 + (ok ? key : 0)) * ld_qkv;
      cp_async16(smem_u32(kd + swz(r, c, DH)), qkv + row + kcol + c, ok);
      cp_async16(smem_u32(vd + swz(r, c, DH)), qkv + row + vcol + c, ok);
    }
  };
  load_kv(0, 0);
  cp_commit();

  uint32_t qf[DH / 16][4];
  float o[DH / 8][4];
#pragma unroll
  for (int i = 0; i < DH / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_r[2] = {-INFINITY, -INFINITY}, l_r[2] = {0.f, 0.f};
  const int g = lane >> 2, t4 = lane & 3;
  const int qrow0 = q0 + warp * 16 + g;  // rows qrow0 and qrow0 + 8 (sequence-local)

  for (int kt = 0; kt < n_kt; ++kt) {
    if (kt + 1 < n_kt) {
      load_kv(kt + 1, (kt + 1) & 1);
      cp_commit();
      cp_wait<1>();
    } else {
      cp_wait<0>();
    }
    __syncthreads();
    if (kt == 0) {
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk) {
        const int r = warp * 16 + (lane & 15), c = kk * 16 + (lane >> 4) * 8;
        ldsm_x4(smem_u32(Qs + swz(r, c, DH)), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
      }
    }
    const __nv_bfloat16* kb = Ks + (kt & 1) * BKV * DH;
    const __nv_bfloat16* vb = Vs + (kt & 1) * BKV * DH;

    float s[BKV / 8][4];
#pragma unroll
    for (int i = 0; i < BKV / 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < DH / 16; ++kk) {
#pragma unroll
      for (int np = 0; np < BKV / 16; ++np) {
        const int key = np * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int c = kk * 16 + ((lane >> 3) & 1) * 8;
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(kb + swz(key, c, DH)), b0, b1, b2, b3);
        mma16816(s[2 * np], qf[kk], b0, b1);
        mma16816(s[2 * np + 1], qf[kk], b2, b3);
      }
    }
    // mask + online softmax (rows g and g + 8 of this warp)
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int nt = 0; nt < BKV / 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kt * BKV + nt * 8 + 2 * t4 + (e & 1);
        const int qr = qrow0 + (e >> 1) * 8;
        if (key >= len || (causal && key > qr)) s[nt][e] = -INFINITY;
        mx[e >> 1] = fmaxf(mx[e >> 1], s[nt][e]);
      }
    }
    float corr[2], mnew[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
      mnew[r] = fmaxf(m_r[r], mx[r]);
      corr[r] = (m_r[r] == -INFINITY) ? 0.f : exp2f((m_r[r] - mnew[r]) * scale_log2);
      m_r[r] = mnew[r];
      l_r[r] *= corr[r];
    }
#pragma unroll
    for (int i = 0; i < DH / 8; ++i) {
      o[i][0] *= corr[0]; o[i][1] *= corr[0];
      o[i][2] *= corr[1]; o[i][3] *= corr[1];
    }
    // P as a bf16 pair hi + lo (hi = bf16(p), lo = bf16(p - hi)): the P V product
    // then carries ~16 mantissa bits of P instead of 8, for twice the (small) P V work
    uint32_t pa[BKV / 16][4], pl[BKV / 16][4];
#pragma unroll
    for (int nt = 0; nt < BKV / 8; ++nt) {
      float p[4], r[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float mm = mnew[e >> 1];
        p[e] = (s[nt][e] == -INFINITY) ? 0.f : exp2f((s[nt][e] - mm) * scale_log2);
        l_r[e >> 1] += p[e];
      }
      const uint32_t h01 = pack_bf16x2(p[0], p[1]), h23 = pack_bf16x2(p[2], p[3]);
      const float2 f01 = unpack_bf16x2(h01), f23 = unpack_bf16x2(h23);
      r[0] = p[0] - f01.x; r[1] = p[1] - f01.y; r[2] = p[2] - f23.x; r[3] = p[3] - f23.y;
      pa[nt >> 1][(nt & 1) * 2 + 0] = h01;
      pa[nt >> 1][(nt & 1) * 2 + 1] = h23;
      pl[nt >> 1][(nt & 1) * 2 + 0] = pack_bf16x2(r[0], r[1]);
      pl[nt >> 1][(nt & 1) * 2 + 1] = pack_bf16x2(r[2], r[3]);
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < BKV / 16; ++kk) {
      const uint32_t a[4] = {pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3]};
      const uint32_t al[4] = {pl[kk][0], pl[kk][1], pl[kk][2], pl[kk][3]};
#pragma unroll
      for (int nd = 0; nd < DH / 16; ++nd) {
        const int key = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int c = nd * 16 + (lane >> 4) * 8;
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(smem_u32(vb + swz(key, c, DH)), b0, b1, b2, b3);
        mma16816(o[2 * nd], a, b0, b1);
        mma16816(o[2 * nd + 1], a, b2, b3);
        mma16816(o[2 * nd], al, b0, b1);
        mma16816(o[2 * nd + 1], al, b2, b3);
      }
    }
    __syncthreads();
  }

#pragma unroll
  for (int r = 0; r < 2; ++r) {
    l_r[r] += __shfl_xor_sync(0xffffffffu, l_r[r], 1);
    l_r[r] += __shfl_xor_sync(0xffffffffu, l_r[r], 2);
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int qr = qrow0 + r * 8;
    if (qr >= len) continue;
    const float inv = 1.f / l_r[r];
    __nv_bfloat16* dst = out + (size_t)(s0 + qr) * ld_out + h * DH + 2 * t4;
#pragma unroll
    for (int nt = 0; nt < DH / 8; ++nt) {
      *reinterpret_cast<uint32_t*>(dst + nt * 8) =
          pack_bf16x2(o[nt][2 * r] * inv, o[nt][2 * r + 1] * inv);
    }
  }
}

}  // namespace

cudaError_t attention_varlen(const void* qkv, void* out, const int* cu_seqlens, int B,
                             int max_seqlen_cap, int Hq, int Hkv, int dh, bool causal,
                             cudaStream_t st) {
  if (B <= 0 || max_seqlen_cap <= 0) return cudaSuccess;
  dim3 grid((max_seqlen_cap + BQ - 1) / BQ, Hq, B);
  const int ld_qkv = (Hq + 2 * Hkv) * dh, ld_out = Hq * dh;
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)dh);
  const size_t smem = (size_t)(BQ + 4 * BKV) * dh * 2;
  prof_begin_launch(st);
  cudaError_t r;
  if (dh == 128) {
    static bool attr = false;
    if (!attr) {
      r = cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (r != cudaSuccess) return r;
      attr = true;
    }
    attn_kernel<128><<<grid, 128, smem, st>>>(reinterpret_cast<const __nv_bfloat16*>(qkv),
                                              reinterpret_cast<__nv_bfloat16*>(out), cu_seqlens, Hq, Hkv,
                                              ld_qkv, ld_out, causal ? 1 : 0, scale_log2);
  } else if (dh == 64) {
    static bool attr = false;
    if (!attr) {
      r = cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (r != cudaSuccess) return r;
      attr = true;
    }
    attn_kernel<64><<<grid, 128, smem, st>>>(reinterpret_cast<const __nv_bfloat16*>(qkv),
                                             reinterpret_cast<__nv_bfloat16*>(out), cu_seqlens, Hq, Hkv,
                                             ld_qkv, ld_out, causal ? 1 : 0, scale_log2);
  } else {
    return cudaErrorInvalidValue;
  }
  prof_end_launch(st, SP_K_ATTN, 0.0, 0.0);
  return cudaGetLastError();
}

}  // namespace sp
