// Candidate precompute support (Sec. 3.2, the pointer decoder's per-candidate
// rows): the set-up fold of the decoder matrices, and the fp32 operand split
// that lets the bf16 tensor-core GEMM compute the fp32 precompute products.
//
// The selection loop compares pointer logits to 1e-4, so the rows it reads
// (decoder tokens, folded keys / queries / values of every candidate) need
// fp32 accuracy.  An fp32 value x splits exactly-enough into three bf16 parts
// x = x0 + x1 + x2 + r (x0 = bf16(x), x1 = bf16(x - x0), x2 = bf16(x - x0 - x1),
// |r| <= 2^-24 |x| roughly, the residuals being exact in fp32), and
//   a . b ~= a0.b0 + a0.b1 + a1.b0 + a0.b2 + a1.b1 + a2.b0
// keeps every product down to relative weight 2^-16 * 2^-8 (the three dropped
// ones are below 2^-24).  As one GEMM over a K six times longer:
//   A segments [a0 a0 a1 a0 a1 a2]  x  B segments [b0 b1 b0 b2 b1 b0],
// with fp32 accumulation in TMEM.  A is stored once as [a0 a1 a2] (3K wide) and
// the GEMM producer maps each K segment to its part (GemmASplit); the weight
// side is expanded to 6K once, at selector creation.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

SP_DEVINL void split3(float x, __nv_bfloat16& p0, __nv_bfloat16& p1, __nv_bfloat16& p2) {
  p0 = __float2bfloat16_rn(x);
  const float r1 = x - __bfloat162float(p0);
  p1 = __float2bfloat16_rn(r1);
  const float r2 = r1 - __bfloat162float(p1);
  p2 = __float2bfloat16_rn(r2);
}

// out[r, s*K + k] = part s of x[r, k], s = 0, 1, 2 (4 elements per thread).
__global__ void split3_kernel(const float* __restrict__ x, int ldx, int rows, int K, __nv_bfloat16* __restrict__ out) {
  const int q = K >> 2;
  const long long n = (long long)rows * q;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
    const int r = (int)(i / q), k = (int)(i - (long long)r * q) * 4;
    const float4 v = *reinterpret_cast<const float4*>(x + (size_t)r * ldx + k);
    __nv_bfloat16 a[3][4];
    split3(v.x, a[0][0], a[1][0], a[2][0]);
    split3(v.y, a[0][1], a[1][1], a[2][1]);
    split3(v.z, a[0][2], a[1][2], a[2][2]);
    split3(v.w, a[0][3], a[1][3], a[2][3]);
    __nv_bfloat16* o = out + (size_t)r * 3 * K + k;
#pragma unroll
    for (int s = 0; s < 3; ++s) *reinterpret_cast<uint2*>(o + (size_t)s * K) = *reinterpret_cast<const uint2*>(a[s]);
  }
}

// out[n, s*K + k] = part pat[s] of w[n, k] for the six weight segments.
__global__ void split6_weights_kernel(const float* __restrict__ w, int N, int K, __nv_bfloat16* __restrict__ out) {
  const long long n = (long long)N * K;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
    const int r = (int)(i / K), k = (int)(i - (long long)r * K);
    __nv_bfloat16 p[3];
    split3(w[i], p[0], p[1], p[2]);
    const int pat[6] = {0, 1, 0, 2, 1, 0};
    __nv_bfloat16* o = out + (size_t)r * 6 * K + k;
#pragma unroll
    for (int s = 0; s < 6; ++s) o[(size_t)s * K] = p[pat[s]];
  }
}

__global__ void fold_kernel(const float* __restrict__ A, long sai, long sak, const float* __restrict__ B,
                            long sbk, long sbj, float* __restrict__ C, int ldc, int I, int J, int K,
                            float scale) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  const int i = blockIdx.y;
  if (i >= I || j >= J) return;
  double s = 0.0;
  for (int k = 0; k < K; ++k) s += (double)A[i * sai + k * sak] * (double)B[k * sbk + j * sbj];
  C[(size_t)i * ldc + j] = (float)(s * (double)scale);
}

}  // namespace

// A-side segment map of the split product: segments a0 a0 a1 a0 a1 a2.
GemmASplit split3_a_map(int K) {
  GemmASplit s;
  s.seg = K;
  s.map = (0u << 0) | (0u << 4) | (1u << 8) | (0u << 12) | (1u << 16) | (2u << 20);
  return s;
}

cudaError_t split3_bf16(const float* x, int ldx, int rows, int K, void* out, cudaStream_t st) {
  if (rows <= 0) return cudaSuccess;
  if (K % 4 != 0 || ldx % 4 != 0) return cudaErrorInvalidValue;
  const long long n = (long long)rows * (K / 4);
  const int grid = (int)std::min<long long>((n + 255) / 256, (long long)device_sm_count() * 16);
  prof_begin_launch(st);
  split3_kernel<<<grid, 256, 0, st>>>(x, ldx, rows, K, reinterpret_cast<__nv_bfloat16*>(out));
  prof_end_launch(st, SP_K_SGEMM, 0.0, (double)rows * K * (4.0 + 6.0));
  return cudaGetLastError();
}

cudaError_t split6_weights(const float* w, int N, int K, void* out, cudaStream_t st) {
  const long long n = (long long)N * K;
  if (n <= 0) return cudaSuccess;
  const int grid = (int)std::min<long long>((n + 255) / 256, 4096);
  split6_weights_kernel<<<grid, 256, 0, st>>>(w, N, K, reinterpret_cast<__nv_bfloat16*>(out));
  return cudaGetLastError();
}

cudaError_t fold_matmul(const float* A, long sai, long sak, const float* B, long sbk, long sbj,
                        float* C, int ldc, int I, int J, int K, float scale, cudaStream_t st) {
  dim3 grid((J + 127) / 128, I);
  fold_kernel<<<grid, 128, 0, st>>>(A, sai, sak, B, sbk, sbj, C, ldc, I, J, K, scale);
  return cudaGetLastError();
}

}  // namespace sp
