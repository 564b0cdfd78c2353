// Row-wise kernels: RMSNorm (LM), LayerNorm (selector), dtype conversion and the
// small layout kernels that build the encoder input and the candidate memory.
// All are HBM-bound: one block per row, the row held in registers/shared
// memory, one read and one write of it.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

constexpr int NT = 256;

SP_DEVINL float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = (l < (int)(blockDim.x >> 5)) ? red[l] : 0.f;
  t = warp_sum(t);
  return t;
}

SP_DEVINL int rows_from(int rows_cap, const int* row_count) {
  int r = rows_cap;
  if (row_count) r = min(r, __ldg(row_count));
  return r;
}

// d multiple of 4
template <bool OUT_BF16>
__global__ void __launch_bounds__(NT)
rmsnorm_kernel(const float* __restrict__ x, const float* __restrict__ gain, void* __restrict__ out,
               int rows_cap, const int* __restrict__ row_count, int d, float eps) {
  __shared__ float red[32];
  pdl_wait();
  pdl_trigger();
  const int row = blockIdx.x;
  if (row >= rows_from(rows_cap, row_count)) return;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)row * d);
  const int n4 = d >> 2;
  float ss = 0.f;
  for (int i = threadIdx.x; i < n4; i += NT) {
    const float4 v = xr[i];
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = block_sum(ss, red);
  const float r = rsqrtf(ss / (float)d + eps);
  for (int i = threadIdx.x; i < n4; i += NT) {
    float4 v = xr[i];
    float4 g = gain ? reinterpret_cast<const float4*>(gain)[i] : make_float4(1.f, 1.f, 1.f, 1.f);
    v.x *= r * g.x; v.y *= r * g.y; v.z *= r * g.z; v.w *= r * g.w;
    if (OUT_BF16) {
      uint2 u;
      u.x = pack_bf16x2(v.x, v.y);
      u.y = pack_bf16x2(v.z, v.w);
      reinterpret_cast<uint2*>(out)[(size_t)row * n4 + i] = u;
    } else {
      reinterpret_cast<float4*>(out)[(size_t)row * n4 + i] = v;
    }
  }
}

// LayerNorm of fp32 rows (ldx apart) into fp32 and/or bf16 rows (ldo apart), times `scale`.
__global__ void __launch_bounds__(NT)
layernorm_kernel(const float* __restrict__ x, int ldx, const float* __restrict__ gain,
                 const float* __restrict__ bias, float* __restrict__ out_f32, void* __restrict__ out_bf16,
                 int ldo, int rows, int d, float eps, float scale) {
  extern __shared__ float buf[];
  __shared__ float red[32];
  const int row = blockIdx.x;
  if (row >= rows) return;
  const float* xr = x + (size_t)row * ldx;
  float s = 0.f;
  for (int i = threadIdx.x; i < d; i += NT) {
    const float v = xr[i];
    buf[i] = v;
    s += v;
  }
  const float mean = block_sum(s, red) / (float)d;
  float q = 0.f;
  for (int i = threadIdx.x; i < d; i += NT) {
    const float c = buf[i] - mean;
    q += c * c;
  }
  const float rstd = rsqrtf(block_sum(q, red) / (float)d + eps);
  for (int i = threadIdx.x; i < d; i += NT) {
    float v = (buf[i] - mean) * rstd;
    if (gain) v *= gain[i];
    if (bias) v += bias[i];
    v *= scale;
    if (out_f32) out_f32[(size_t)row * ldo + i] = v;
    if (out_bf16) reinterpret_cast<__nv_bfloat16*>(out_bf16)[(size_t)row * ldo + i] = __float2bfloat16_rn(v);
  }
}

__global__ void bf16_to_f32_kernel(const uint2* __restrict__ x, float4* __restrict__ out, int rows_cap,
                                   const int* __restrict__ row_count, int d) {
  pdl_wait();
  pdl_trigger();
  const int row = blockIdx.x;
  if (row >= rows_from(rows_cap, row_count)) return;
  const int n4 = d >> 2;
  for (int i = threadIdx.x; i < n4; i += blockDim.x) {
    const uint2 u = x[(size_t)row * n4 + i];
    const float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y);
    out[(size_t)row * n4 + i] = make_float4(a.x, a.y, b.x, b.y);
  }
}

// Rows [T, T + gridDim.x) of a row-major buffer, T = *row_count, below rows_cap, set to zero.
__global__ void zero_rows_after_kernel(uint4* __restrict__ buf, int row_u4, const int* __restrict__ row_count,
                                       int rows_cap) {
  pdl_wait();
  pdl_trigger();
  const int row = __ldg(row_count) + blockIdx.x;
  if (row < 0 || row >= rows_cap) return;
  for (int i = threadIdx.x; i < row_u4; i += blockDim.x) buf[(size_t)row * row_u4 + i] = make_uint4(0, 0, 0, 0);
}

SP_DEVINL int find_image(const int* off, int B, int r) {
  // largest b with off[b] <= r
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= r) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Encoder input rows of image b: [X_b (bf16 -> fp32); g_text * LN(P_b)] (Eq. 3).
__global__ void __launch_bounds__(NT)
assemble_kernel(const BatchDesc bd, const __nv_bfloat16* __restrict__ X, const float* __restrict__ P,
                int D, const float* __restrict__ g, const float* __restrict__ bb, float eps,
                float g_text, float* __restrict__ R, int rows) {
  extern __shared__ float buf[];
  __shared__ float red[32];
  const int r = blockIdx.x;
  if (r >= rows) return;
  int enc_off[1];
  // enc_off[b] = vis_off[b] + txt_off[b]; binary search on it
  int lo = 0, hi = bd.B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (bd.vis_off[mid] + bd.txt_off[mid] <= r) lo = mid; else hi = mid - 1;
  }
  const int b = lo;
  enc_off[0] = bd.vis_off[b] + bd.txt_off[b];
  const int local = r - enc_off[0];
  const int nv = bd.vis_off[b + 1] - bd.vis_off[b];
  float* out = R + (size_t)r * D;
  if (local < nv) {
    const __nv_bfloat16* xr = X + (size_t)(bd.vis_off[b] + local) * D;
    for (int i = threadIdx.x; i < D; i += NT) out[i] = __bfloat162float(xr[i]);
    return;
  }
  const float* pr = P + (size_t)(bd.txt_off[b] + local - nv) * D;
  float s = 0.f;
  for (int i = threadIdx.x; i < D; i += NT) {
    const float v = pr[i];
    buf[i] = v;
    s += v;
  }
  const float mean = block_sum(s, red) / (float)D;
  float q = 0.f;
  for (int i = threadIdx.x; i < D; i += NT) {
    const float c = buf[i] - mean;
    q += c * c;
  }
  const float rstd = rsqrtf(block_sum(q, red) / (float)D + eps);
  for (int i = threadIdx.x; i < D; i += NT) {
    float v = (buf[i] - mean) * rstd;
    if (g) v *= g[i];
    if (bb) v += bb[i];
    out[i] = g_text * v;
  }
}

// Candidate memory rows: [H (every image's visual rows); s_stop; s_start].
__global__ void gather_memory_kernel(const BatchDesc bd, const float* __restrict__ R,
                                     const float* __restrict__ H, const float* __restrict__ s_stop,
                                     const float* __restrict__ s_start, float* __restrict__ Mall, int D) {
  const int r = blockIdx.x;
  const int nvis = bd.vis_off[bd.B];
  const float* src;
  if (r < nvis) {
    if (H) {
      src = H + (size_t)r * D;
    } else {
      const int b = find_image(bd.vis_off, bd.B, r);
      const int enc_row = bd.vis_off[b] + bd.txt_off[b] + (r - bd.vis_off[b]);
      src = R + (size_t)enc_row * D;
    }
  } else {
    src = (r == nvis) ? s_stop : s_start;
  }
  for (int i = threadIdx.x; i < D; i += blockDim.x) Mall[(size_t)r * D + i] = src[i];
}

__global__ void write_enc_cu_kernel(const BatchDesc bd, int* cu) {
  for (int b = threadIdx.x; b <= bd.B; b += blockDim.x) cu[b] = bd.vis_off[b] + bd.txt_off[b];
}

}  // namespace

cudaError_t rmsnorm_f32_to_bf16(const float* x, const float* gain, void* out, int rows_cap,
                                const int* row_count, int d, float eps, cudaStream_t st) {
  if (rows_cap <= 0) return cudaSuccess;
  prof_begin_launch(st);
  const cudaError_t r = launch_pdl(rmsnorm_kernel<true>, dim3(rows_cap), dim3(NT), 0, st, x, gain, out, rows_cap,
                                   row_count, d, eps);
  prof_end_launch(st, SP_K_NORM, 0.0, 6.0 * rows_cap * (double)d);
  return r;
}

cudaError_t rmsnorm_f32_to_f32(const float* x, const float* gain, float* out, int rows_cap,
                               const int* row_count, int d, float eps, cudaStream_t st) {
  if (rows_cap <= 0) return cudaSuccess;
  prof_begin_launch(st);
  const cudaError_t r = launch_pdl(rmsnorm_kernel<false>, dim3(rows_cap), dim3(NT), 0, st, x, gain,
                                   static_cast<void*>(out), rows_cap, row_count, d, eps);
  prof_end_launch(st, SP_K_NORM, 0.0, 8.0 * rows_cap * (double)d);
  return r;
}

cudaError_t layernorm_f32(const float* x, int ldx, const float* gain, const float* bias, float* out_f32,
                          void* out_bf16, int ldo, int rows, int d, float eps, float scale,
                          cudaStream_t st) {
  if (rows <= 0) return cudaSuccess;
  prof_begin_launch(st);
  layernorm_kernel<<<rows, NT, d * sizeof(float), st>>>(x, ldx, gain, bias, out_f32, out_bf16, ldo, rows,
                                                        d, eps, scale);
  prof_end_launch(st, SP_K_NORM, 0.0, 6.0 * rows * (double)d);
  return cudaGetLastError();
}

cudaError_t zero_rows_after(void* buf, size_t row_bytes, const int* row_count, int rows_cap, int nrows,
                            cudaStream_t st) {
  if (rows_cap <= 0 || nrows <= 0) return cudaSuccess;
  if (row_bytes % 16 != 0) return cudaErrorInvalidValue;
  prof_begin_launch(st);
  const cudaError_t r = launch_pdl(zero_rows_after_kernel, dim3(nrows), dim3(256), 0, st,
                                   reinterpret_cast<uint4*>(buf), (int)(row_bytes / 16), row_count, rows_cap);
  prof_end_launch(st, SP_K_MISC, 0.0, (double)nrows * row_bytes);
  return r;
}

cudaError_t bf16_to_f32(const void* x, float* out, int rows_cap, const int* row_count, int d,
                        cudaStream_t st) {
  if (rows_cap <= 0) return cudaSuccess;
  prof_begin_launch(st);
  const cudaError_t r = launch_pdl(bf16_to_f32_kernel, dim3(rows_cap), dim3(256), 0, st,
                                   reinterpret_cast<const uint2*>(x), reinterpret_cast<float4*>(out), rows_cap,
                                   row_count, d);
  prof_end_launch(st, SP_K_MISC, 0.0, 6.0 * rows_cap * (double)d);
  return r;
}

cudaError_t assemble_encoder_input(const BatchDesc& bd, const void* X, const float* P, int D,
                                   const float* ln_g, const float* ln_b, float eps, float g_text,
                                   float* R, int rows, cudaStream_t st) {
  if (rows <= 0) return cudaSuccess;
  prof_begin_launch(st);
  assemble_kernel<<<rows, NT, D * sizeof(float), st>>>(bd, reinterpret_cast<const __nv_bfloat16*>(X), P,
                                                       D, ln_g, ln_b, eps, g_text, R, rows);
  prof_end_launch(st, SP_K_MISC, 0.0, 6.0 * rows * (double)D);
  return cudaGetLastError();
}

cudaError_t gather_memory(const BatchDesc& bd, const float* R, const float* H, const float* s_stop,
                          const float* s_start, float* Mall, int D, cudaStream_t st) {
  const int rows = bd.vis_off[bd.B] + 2;
  prof_begin_launch(st);
  gather_memory_kernel<<<rows, 256, 0, st>>>(bd, R, H, s_stop, s_start, Mall, D);
  prof_end_launch(st, SP_K_MISC, 0.0, 8.0 * rows * (double)D);
  return cudaGetLastError();
}

cudaError_t write_enc_cu(const BatchDesc& bd, int* cu, cudaStream_t st) {
  write_enc_cu_kernel<<<1, 256, 0, st>>>(bd, cu);
  return cudaGetLastError();
}

}  // namespace sp
