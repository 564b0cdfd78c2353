// Training-time continuous pathway, forward only (Sec. 3.3): the SoftTopK
// polarisation of the trajectory scores (Eq. 8) and the variance-preserving
// noise gate (Eq. 9).  The scores and soft counts themselves (Eqs. 5-7) are
// accumulated by the selection kernel along the rollout.
//
// SoftTopK_{k,tau}(s) is read as the entropic optimal transport of the n scores
// (mass 1/n each) onto two anchors y = (0, 1) with masses ((n - k)/n, k/n),
// cost (s_i - y_j)^2 and regularisation tau, alpha_i = n Gamma_i,2.  With two
// anchors the optimal plan's row ratio Gamma_i,2 / Gamma_i,1 is
// exp((2 s_i - 1 + g_2 - g_1) / tau), so alpha_i = sigmoid(2 (s_i - theta) / tau)
// where theta is the one value with sum_i alpha_i = k.  The kernel finds theta
// directly: sum_i alpha_i is strictly decreasing in theta, so a bracket is
// shrunk nine-fold per step (eight warps evaluate eight interior points at once)
// until it stops shrinking in fp32.  No Sinkhorn iterations, whose convergence
// slows down when tau is small against the spread of the scores.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

constexpr int TK_NT = 256;
constexpr int TK_NW = TK_NT / 32;
constexpr int TK_STEPS = 24;

SP_DEVINL float sigmoidf(float z) { return 1.f / (1.f + expf(-z)); }

// Block-wide sum of one value per thread; every thread gets the total, summed
// in warp order (red: TK_NW floats; ends with a barrier so red can be reused).
SP_DEVINL float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) red[w] = v;
  __syncthreads();
  float t = 0.f;
#pragma unroll
  for (int k = 0; k < TK_NW; ++k) t += red[k];
  __syncthreads();
  return t;
}

SP_DEVINL float block_min_max(float v, float* red, bool is_max) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float u = __shfl_xor_sync(0xffffffffu, v, o);
    v = is_max ? fmaxf(v, u) : fminf(v, u);
  }
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) red[w] = v;
  __syncthreads();
  float t = red[0];
#pragma unroll
  for (int k = 1; k < TK_NW; ++k) t = is_max ? fmaxf(t, red[k]) : fminf(t, red[k]);
  __syncthreads();
  return t;
}

// One CTA per image.  k = (sum of every episode's soft count) / B: the batch
// mean of the images' soft counts (each image's count is the sum over its
// episodes), detached; clamped to [0, N_b] per image.
__global__ void __launch_bounds__(TK_NT)
soft_topk_kernel(const BatchDesc bd, int n_episodes, const float* __restrict__ score, const float* __restrict__ kbar,
                 float two_over_tau, float* __restrict__ alpha, float* __restrict__ k_out) {
  extern __shared__ float s_sc[];
  __shared__ float red[TK_NW];
  __shared__ float fval[TK_NW];
  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int v0 = bd.vis_off[b], n = bd.vis_off[b + 1] - v0;

  float part = 0.f;
  for (int e = tid; e < n_episodes; e += TK_NT) part += kbar[e];
  const float k_mean = block_sum(part, red) / (float)bd.B;
  if (b == 0 && tid == 0 && k_out) *k_out = k_mean;
  const float k = fminf(fmaxf(k_mean, 0.f), (float)n);
  if (n == 0) return;
  if (!(k > 0.f) || k >= (float)n) {  // the plan is fixed by the marginals
    const float v = k >= (float)n ? 1.f : 0.f;
    for (int i = tid; i < n; i += TK_NT) alpha[v0 + i] = v;
    return;
  }
  float lo_v = INFINITY, hi_v = -INFINITY;
  for (int i = tid; i < n; i += TK_NT) {
    const float x = score[v0 + i];
    s_sc[i] = x;
    lo_v = fminf(lo_v, x);
    hi_v = fmaxf(hi_v, x);
  }
  lo_v = block_min_max(lo_v, red, false);
  hi_v = block_min_max(hi_v, red, true);
  // sum alpha > k at lo (every sigmoid ~ 1), < k at hi (every sigmoid ~ 0)
  float lo = lo_v - 24.f / two_over_tau, hi = hi_v + 24.f / two_over_tau;
  for (int step = 0; step < TK_STEPS; ++step) {
    const float th = lo + (hi - lo) * (float)(warp + 1) / (float)(TK_NW + 1);
    float f = 0.f;
    for (int i = lane; i < n; i += 32) f += sigmoidf((s_sc[i] - th) * two_over_tau);
    f = warp_sum(f);
    if (lane == 0) fval[warp] = f - k;
    __syncthreads();
    // first interior point where the sum has fallen below k (identical in every thread)
    float nlo = lo, nhi = hi;
    for (int w = 0; w < TK_NW; ++w) {
      const float tw = lo + (hi - lo) * (float)(w + 1) / (float)(TK_NW + 1);
      if (fval[w] > 0.f) {
        nlo = tw;
      } else {
        nhi = tw;
        break;
      }
    }
    __syncthreads();
    if (nlo == lo && nhi == hi) break;  // no interior point left in fp32
    lo = nlo;
    hi = nhi;
  }
  const float theta = 0.5f * (lo + hi);
  for (int i = tid; i < n; i += TK_NT) alpha[v0 + i] = sigmoidf((s_sc[i] - theta) * two_over_tau);
}

// Eq. 9 on 8 bf16 per thread-iteration: out = sqrt(alpha_r) x + sqrt(1 - alpha_r) eps.
__global__ void __launch_bounds__(256)
vp_gate_kernel(const uint4* __restrict__ X, const uint4* __restrict__ noise, const float* __restrict__ alpha,
               uint4* __restrict__ out, long long chunks, int chunks_per_row) {
  for (long long c = blockIdx.x * (long long)blockDim.x + threadIdx.x; c < chunks;
       c += (long long)gridDim.x * blockDim.x) {
    const int r = (int)(c / chunks_per_row);
    const float a = fminf(fmaxf(__ldg(alpha + r), 0.f), 1.f);
    const float sa = sqrtf(a), sb = sqrtf(1.f - a);
    const uint4 x = __ldg(X + c), e = __ldg(noise + c);
    const uint32_t xs[4] = {x.x, x.y, x.z, x.w}, es[4] = {e.x, e.y, e.z, e.w};
    uint32_t o[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 xv = unpack_bf16x2(xs[q]), ev = unpack_bf16x2(es[q]);
      o[q] = pack_bf16x2(sa * xv.x + sb * ev.x, sa * xv.y + sb * ev.y);
    }
    out[c] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

}  // namespace

cudaError_t soft_topk_launch(const BatchDesc& bd, int n_episodes, const float* score, const float* kbar, float tau,
                             float* alpha, float* k_out, cudaStream_t st) {
  int n_max = 0;
  for (int b = 0; b < bd.B; ++b) n_max = std::max(n_max, bd.vis_off[b + 1] - bd.vis_off[b]);
  const size_t smem = (size_t)std::max(n_max, 1) * sizeof(float);
  if (smem > 48 * 1024) {
    cudaError_t r = cudaFuncSetAttribute(soft_topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (r != cudaSuccess) return r;
  }
  prof_begin_launch(st);
  soft_topk_kernel<<<bd.B, TK_NT, smem, st>>>(bd, n_episodes, score, kbar, 2.f / tau, alpha, k_out);
  prof_end_launch(st, SP_K_TRAIN, 0.0, 0.0);
  return cudaGetLastError();
}

cudaError_t vp_gate_launch(const void* X, const void* noise, const float* alpha, void* out, int rows, int D,
                           cudaStream_t st) {
  const long long chunks = (long long)rows * (D / 8);
  if (chunks == 0) return cudaSuccess;
  const int sms = device_sm_count();
  const long long want = (chunks + 255) / 256;
  const int grid = (int)std::min<long long>(want, (long long)sms * 8);
  prof_begin_launch(st);
  vp_gate_kernel<<<grid, 256, 0, st>>>(reinterpret_cast<const uint4*>(X), reinterpret_cast<const uint4*>(noise),
                                       alpha, reinterpret_cast<uint4*>(out), chunks, D / 8);
  prof_end_launch(st, SP_K_TRAIN, 0.0, (double)chunks * 48.0);
  return cudaGetLastError();
}

}  // namespace sp
