// The key / value cache and the generation step that follows the prefill
// over the pruned prefix: the prefill writes every packed row's rotated key
// and value into a per-sequence cache; a decode step appends one token per
// sequence and attends over that sequence's cache.
//
// Cache layout (bf16), per layer l, sequence b, position p:
//   K at ((l * 2 + 0) * B + b) * S_cap + p rows of W = Hkv * dh elements,
//   V at ((l * 2 + 1) * B + b) * S_cap + p.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

// Copy one row of n16 16-byte chunks, eight in flight per lane.
SP_DEVINL void copy16(const uint4* __restrict__ src, uint4* __restrict__ dst, int n16, int lane) {
  for (int i = lane; i < n16; i += 8 * 32) {
    uint4 v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (i + u * 32 < n16) v[u] = __ldg(src + i + u * 32);
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (i + u * 32 < n16) dst[i + u * 32] = v[u];
  }
}

// Prefill rows -> cache: one warp per packed row (K and V of all kv heads).
__global__ void __launch_bounds__(256) kv_store_kernel(const __nv_bfloat16* __restrict__ qkv, int ld_qkv,
                                                       int kcol, int vcol, int W, const int* __restrict__ cu,
                                                       const int* __restrict__ pos, int B, int T_cap,
                                                       __nv_bfloat16* __restrict__ kv_l, int S_cap, int* err) {
  __shared__ int s_cu[SP_MAX_BATCH + 1];
  pdl_wait();
  pdl_trigger();
  for (int i = threadIdx.x; i <= B; i += blockDim.x) s_cu[i] = __ldg(cu + i);
  __syncthreads();
  const int T = min(s_cu[B], T_cap);
  const int lane = threadIdx.x & 31;
  const int n16 = W / 8;
  for (int r = blockIdx.x * 8 + (threadIdx.x >> 5); r < T; r += gridDim.x * 8) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (s_cu[mid] <= r) lo = mid; else hi = mid - 1;
    }
    const int p = __ldg(pos + r);
    if (p < 0 || p >= S_cap) {
      if (lane == 0) set_error(err, SP_DEVERR_INDEX);
      continue;
    }
    const __nv_bfloat16* row = qkv + (size_t)r * ld_qkv;
    __nv_bfloat16* kd = kv_l + ((size_t)lo * S_cap + p) * W;
    __nv_bfloat16* vd = kv_l + ((size_t)(B + lo) * S_cap + p) * W;
    copy16(reinterpret_cast<const uint4*>(row + kcol), reinterpret_cast<uint4*>(kd), n16, lane);
    copy16(reinterpret_cast<const uint4*>(row + vcol), reinterpret_cast<uint4*>(vd), n16, lane);
  }
}

// Decode rows -> cache at position lens[b]: one warp per sequence.
__global__ void __launch_bounds__(256) kv_append_kernel(const __nv_bfloat16* __restrict__ qkv, int ld_qkv,
                                                        int kcol, int vcol, int W, const int* __restrict__ lens,
                                                        int B, __nv_bfloat16* __restrict__ kv_l, int S_cap,
                                                        int* err) {
  const int b = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (b >= B) return;
  const int p = __ldg(lens + b);
  if (p < 0 || p >= S_cap) {
    if (lane == 0) set_error(err, SP_DEVERR_INDEX);
    return;
  }
  const __nv_bfloat16* row = qkv + (size_t)b * ld_qkv;
  copy16(reinterpret_cast<const uint4*>(row + kcol), reinterpret_cast<uint4*>(kv_l + ((size_t)b * S_cap + p) * W),
         W / 8, lane);
  copy16(reinterpret_cast<const uint4*>(row + vcol),
         reinterpret_cast<uint4*>(kv_l + ((size_t)(B + b) * S_cap + p) * W), W / 8, lane);
}

// Attention of the new token of sequence b, query head h, over the cached
// positions 0..lens[b] (the new one included).  One CTA per (h, b), 4 warps
// taking 32-key blocks round-robin: in a block lane j scores key j (its whole
// dot product), the warp updates its running max / sum, then accumulates
// P V with lane-owned head dims.  The warps' partials merge in shared memory.
template <int DH>
__global__ void __launch_bounds__(128) decode_attn_kernel(const __nv_bfloat16* __restrict__ qkv, int ld_qkv,
                                                          const __nv_bfloat16* __restrict__ kv_l, int S_cap,
                                                          const int* __restrict__ lens, int B, int Hq, int Hkv,
                                                          __nv_bfloat16* __restrict__ out, int ld_out,
                                                          float scale_log2) {
  constexpr int DPL = DH / 32;  // head dims per lane in P V
  __shared__ __align__(16) float q_s[DH];
  __shared__ float m_s[4], l_s[4];
  __shared__ float o_s[4][DH];
  const int h = blockIdx.x, b = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int W = Hkv * DH;
  const int kvh = h / (Hq / Hkv);
  const int L = min(__ldg(lens + b), S_cap - 1) + 1;  // positions 0..lens[b]
  for (int d = threadIdx.x; d < DH; d += 128) q_s[d] = __bfloat162float(qkv[(size_t)b * ld_qkv + h * DH + d]);
  __syncthreads();
  const __nv_bfloat16* Kb = kv_l + (size_t)b * S_cap * W + kvh * DH;
  const __nv_bfloat16* Vb = kv_l + (size_t)(B + b) * S_cap * W + kvh * DH;
  float m = -INFINITY, l = 0.f, o[DPL];
#pragma unroll
  for (int i = 0; i < DPL; ++i) o[i] = 0.f;
  for (int j0 = warp * 32; j0 < L; j0 += 4 * 32) {
    const int j = j0 + lane;
    float s = -INFINITY;
    if (j < L) {
      const uint4* kr = reinterpret_cast<const uint4*>(Kb + (size_t)j * W);
      float acc = 0.f;
#pragma unroll 4
      for (int c = 0; c < DH / 8; ++c) {
        const uint4 u = __ldg(kr + c);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = unpack_bf16x2(w[e]);
          acc += f.x * q_s[c * 8 + 2 * e] + f.y * q_s[c * 8 + 2 * e + 1];
        }
      }
      s = acc * scale_log2;
    }
    const float mb = warp_max(s);
    const float mn = fmaxf(m, mb);
    const float corr = (m == -INFINITY) ? 0.f : exp2f(m - mn);
    const float p = (j < L) ? exp2f(s - mn) : 0.f;
    l = l * corr + warp_sum(p);
#pragma unroll
    for (int i = 0; i < DPL; ++i) o[i] *= corr;
    const int nk = min(32, L - j0);
    for (int k = 0; k < nk; ++k) {
      const float pk = __shfl_sync(0xffffffffu, p, k);
      const __nv_bfloat16* vr = Vb + (size_t)(j0 + k) * W + lane * DPL;
      if (DPL == 4) {
        const uint2 u = __ldg(reinterpret_cast<const uint2*>(vr));
        const float2 a = unpack_bf16x2(u.x), c = unpack_bf16x2(u.y);
        o[0] += pk * a.x; o[1] += pk * a.y; o[2 % DPL] += pk * c.x; o[3 % DPL] += pk * c.y;
      } else {
        const float2 a = unpack_bf16x2(__ldg(reinterpret_cast<const uint32_t*>(vr)));
        o[0] += pk * a.x; o[1 % DPL] += pk * a.y;
      }
    }
    m = mn;
  }
  if (lane == 0) { m_s[warp] = m; l_s[warp] = l; }
#pragma unroll
  for (int i = 0; i < DPL; ++i) o_s[warp][lane * DPL + i] = o[i];
  __syncthreads();
  for (int d = threadIdx.x; d < DH; d += 128) {
    float mm = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) mm = fmaxf(mm, m_s[w]);
    float num = 0.f, den = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float c = (m_s[w] == -INFINITY) ? 0.f : exp2f(m_s[w] - mm);
      num += c * o_s[w][d];
      den += c * l_s[w];
    }
    out[(size_t)b * ld_out + h * DH + d] = __float2bfloat16_rn(num / den);
  }
}

__global__ void lens_increment_kernel(int* lens, int* rope_pos, int B, int S_cap) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B && lens[b] < S_cap) {
    lens[b] += 1;
    if (rope_pos) rope_pos[b] += 1;
  }
}

}  // namespace

cudaError_t kv_store(const void* qkv, const int* cu, const int* pos, int B, int T_cap, int Hq, int Hkv, int dh,
                     void* kv_l, int S_cap, int* err, cudaStream_t st) {
  if (T_cap <= 0) return cudaSuccess;
  const int ld = (Hq + 2 * Hkv) * dh;
  const int grid = std::max(1, std::min((T_cap + 7) / 8, device_sm_count() * 8));
  prof_begin_launch(st);
  const cudaError_t r = launch_pdl(kv_store_kernel, dim3(grid), dim3(256), 0, st,
                                   reinterpret_cast<const __nv_bfloat16*>(qkv), ld, Hq * dh, (Hq + Hkv) * dh, Hkv * dh,
                                   cu, pos, B, T_cap, reinterpret_cast<__nv_bfloat16*>(kv_l), S_cap, err);
  prof_end_launch(st, SP_K_MISC, 0.0, 4.0 * T_cap * Hkv * dh * 2);
  return r;
}

cudaError_t kv_append(const void* qkv, const int* lens, int B, int Hq, int Hkv, int dh, void* kv_l, int S_cap,
                      int* err, cudaStream_t st) {
  const int ld = (Hq + 2 * Hkv) * dh;
  prof_begin_launch(st);
  kv_append_kernel<<<(B + 7) / 8, 256, 0, st>>>(reinterpret_cast<const __nv_bfloat16*>(qkv), ld, Hq * dh,
                                                (Hq + Hkv) * dh, Hkv * dh, lens, B,
                                                reinterpret_cast<__nv_bfloat16*>(kv_l), S_cap, err);
  prof_end_launch(st, SP_K_MISC, 0.0, 4.0 * B * Hkv * dh * 2);
  return cudaGetLastError();
}

cudaError_t decode_attention(const void* qkv, const void* kv_l, int S_cap, const int* lens, int B, int Hq, int Hkv,
                             int dh, void* out, cudaStream_t st) {
  const int ld = (Hq + 2 * Hkv) * dh;
  const float sl2 = 1.4426950408889634f / sqrtf((float)dh);
  dim3 grid(Hq, B);
  prof_begin_launch(st);
  if (dh == 128)
    decode_attn_kernel<128><<<grid, 128, 0, st>>>(reinterpret_cast<const __nv_bfloat16*>(qkv), ld,
                                                   reinterpret_cast<const __nv_bfloat16*>(kv_l), S_cap, lens, B, Hq,
                                                   Hkv, reinterpret_cast<__nv_bfloat16*>(out), Hq * dh, sl2);
  else if (dh == 64)
    decode_attn_kernel<64><<<grid, 128, 0, st>>>(reinterpret_cast<const __nv_bfloat16*>(qkv), ld,
                                                  reinterpret_cast<const __nv_bfloat16*>(kv_l), S_cap, lens, B, Hq,
                                                  Hkv, reinterpret_cast<__nv_bfloat16*>(out), Hq * dh, sl2);
  else
    return cudaErrorInvalidValue;
  prof_end_launch(st, SP_K_ATTN, 0.0, 0.0);
  return cudaGetLastError();
}

cudaError_t lens_increment(int* lens, int* rope_pos, int B, int S_cap, cudaStream_t st) {
  lens_increment_kernel<<<(B + 127) / 128, 128, 0, st>>>(lens, rope_pos, B, S_cap);
  return cudaGetLastError();
}

}  // namespace sp
