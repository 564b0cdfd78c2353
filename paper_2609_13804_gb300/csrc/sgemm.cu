// fp32 SIMT GEMM for the selector's candidate precompute.  The selection loop
// compares pointer logits to 1e-4, so the rows it reads (decoder tokens, folded
// keys/queries/values of every candidate) are computed in fp32 from the fp32
// candidate memory instead of on the bf16 tensor path.
//
// C[M, N] = A[M, K] B[N, K]^T (both operands K-contiguous): 128x128 CTA tile,
// 256 threads each owning an 8x8 block, K in slices of 16 staged transposed in
// shared memory, double-buffered through registers.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

constexpr int TM = 128, TN = 128, TK = 16;

__global__ void __launch_bounds__(256)
sgemm_kernel(const float* __restrict__ A, int lda, const float* __restrict__ B, int ldb,
             float* __restrict__ C, int ldc, int M, int N, int K) {
  __shared__ __align__(16) float As[TK][TM + 4];
  __shared__ __align__(16) float Bs[TK][TN + 4];
  const int tid = threadIdx.x;
  const int tx = tid & 15, ty = tid >> 4;
  const int m0 = blockIdx.y * TM, n0 = blockIdx.x * TN;

  // loader mapping: 128 rows x 16 k = 512 float4 per operand, 2 per thread
  const int lr = tid >> 2;        // 0..63 (+64 for the second)
  const int lk = (tid & 3) * 4;   // 0,4,8,12

  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

  auto load = [&](const float* P, int ld, int rows, int r0, int k0, int r, float4& v) {
    const int gr = r0 + r, gk = k0 + lk;
    v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (gr < rows) {
      const float* p = P + (size_t)gr * ld + gk;
      if (gk + 3 < K && ((reinterpret_cast<uintptr_t>(p) & 15) == 0)) {
        v = *reinterpret_cast<const float4*>(p);
      } else {
        if (gk < K) v.x = p[0];
        if (gk + 1 < K) v.y = p[1];
        if (gk + 2 < K) v.z = p[2];
        if (gk + 3 < K) v.w = p[3];
      }
    }
  };

  float4 ra[2], rb[2];
  for (int i = 0; i < 2; ++i) {
    load(A, lda, M, m0, 0, lr + 64 * i, ra[i]);
    load(B, ldb, N, n0, 0, lr + 64 * i, rb[i]);
  }
  for (int k0 = 0; k0 < K; k0 += TK) {
    __syncthreads();
    for (int i = 0; i < 2; ++i) {
      const int r = lr + 64 * i;
      As[lk + 0][r] = ra[i].x; As[lk + 1][r] = ra[i].y; As[lk + 2][r] = ra[i].z; As[lk + 3][r] = ra[i].w;
      Bs[lk + 0][r] = rb[i].x; Bs[lk + 1][r] = rb[i].y; Bs[lk + 2][r] = rb[i].z; Bs[lk + 3][r] = rb[i].w;
    }
    __syncthreads();
    if (k0 + TK < K) {
      for (int i = 0; i < 2; ++i) {
        load(A, lda, M, m0, k0 + TK, lr + 64 * i, ra[i]);
        load(B, ldb, N, n0, k0 + TK, lr + 64 * i, rb[i]);
      }
    }
#pragma unroll
    for (int k = 0; k < TK; ++k) {
      float a[8], b[8];
      const float4 a0 = *reinterpret_cast<const float4*>(&As[k][ty * 4]);
      const float4 a1 = *reinterpret_cast<const float4*>(&As[k][64 + ty * 4]);
      const float4 b0 = *reinterpret_cast<const float4*>(&Bs[k][tx * 4]);
      const float4 b1 = *reinterpret_cast<const float4*>(&Bs[k][64 + tx * 4]);
      a[0] = a0.x; a[1] = a0.y; a[2] = a0.z; a[3] = a0.w;
      a[4] = a1.x; a[5] = a1.y; a[6] = a1.z; a[7] = a1.w;
      b[0] = b0.x; b[1] = b0.y; b[2] = b0.z; b[3] = b0.w;
      b[4] = b1.x; b[5] = b1.y; b[6] = b1.z; b[7] = b1.w;
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int r = m0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
    if (r >= M) continue;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int c = n0 + (j < 4 ? tx * 4 + j : 64 + tx * 4 + (j - 4));
      if (c < N) C[(size_t)r * ldc + c] = acc[i][j];
    }
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

cudaError_t sgemm_f32(const float* A, int lda, const float* B, int ldb, float* C, int ldc, int M,
                      int N, int K, cudaStream_t st) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  dim3 grid((N + TN - 1) / TN, (M + TM - 1) / TM);
  prof_begin_launch(st);
  sgemm_kernel<<<grid, 256, 0, st>>>(A, lda, B, ldb, C, ldc, M, N, K);
  prof_end_launch(st, SP_K_SGEMM, 2.0 * M * N * (double)K, 4.0 * ((double)M * K + (double)N * K + (double)M * N));
  return cudaGetLastError();
}

cudaError_t fold_matmul(const float* A, long sai, long sak, const float* B, long sbk, long sbj,
                        float* C, int ldc, int I, int J, int K, float scale, cudaStream_t st) {
  dim3 grid((J + 127) / 128, I);
  fold_kernel<<<grid, 128, 0, st>>>(A, sai, sak, B, sbk, sbj, C, ldc, I, J, K, scale);
  return cudaGetLastError();
}

}  // namespace sp
