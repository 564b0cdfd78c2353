// Compaction (Algorithm 1 step 5, X_S = Gather(X, S)): the kept visual rows of
// every image, in native order, followed by its text rows, written as one packed
// variable-length buffer with cu_seqlens and per-sequence positions.  Pure data
// movement, HBM-bound: one warp per output row, 16-byte vector copies.
//
// Every block recomputes the (small) prefix sums of the per-image counts from
// the device counts, so the kernel needs no host round trip and no second
// launch; block 0 publishes cu_seqlens / vis_cu.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

constexpr int NT = 256;

// One row, 16-byte chunks per lane; eight loads are issued before their stores
// so a warp keeps up to 4 KB in flight instead of one chunk per round trip.
SP_DEVINL void copy_row(const uint4* __restrict__ src, uint4* __restrict__ dst, int n16, int lane) {
  int i = lane;
  for (; i + 7 * 32 < n16; i += 8 * 32) {
    uint4 v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = __ldg(src + i + u * 32);
#pragma unroll
    for (int u = 0; u < 8; ++u) dst[i + u * 32] = v[u];
  }
  uint4 v[8];
#pragma unroll
  for (int u = 0; u < 8; ++u)
    if (i + u * 32 < n16) v[u] = __ldg(src + i + u * 32);
#pragma unroll
  for (int u = 0; u < 8; ++u)
    if (i + u * 32 < n16) dst[i + u * 32] = v[u];
}

__global__ void __launch_bounds__(NT, 4)
compact_kernel(const BatchDesc bd, const __nv_bfloat16* __restrict__ X, int W_vis,
               const __nv_bfloat16* __restrict__ text, int W_txt, const int* __restrict__ idx, int k_cap,
               const int* __restrict__ count, __nv_bfloat16* __restrict__ packed, int* __restrict__ cu,
               int* __restrict__ pos, __nv_bfloat16* __restrict__ vis_packed, int* __restrict__ vis_row_map,
               int* __restrict__ vis_cu, int T_cap, int* err) {
  __shared__ int s_cu[SP_MAX_BATCH + 1];
  __shared__ int s_vcu[SP_MAX_BATCH + 1];
  __shared__ int s_cnt[SP_MAX_BATCH];
  __shared__ int wtot[2][NT / 32];
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const int B = bd.B;

  // prefix sums over images (B <= 256 = NT, one image per thread)
  int k = 0, len = 0;
  if (tid < B) {
    const int n_img = bd.vis_off[tid + 1] - bd.vis_off[tid];
    k = __ldg(count + tid);
    if (k < 0 || k > n_img || k > k_cap) {
      set_error(err, SP_DEVERR_INDEX);
      k = max(0, min(k, min(n_img, k_cap)));
    }
    len = k + (bd.txt_off[tid + 1] - bd.txt_off[tid]);
    s_cnt[tid] = k;
  }
  int xk = k, xl = len;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int yk = __shfl_up_sync(0xffffffffu, xk, o);
    const int yl = __shfl_up_sync(0xffffffffu, xl, o);
    if (lane >= o) { xk += yk; xl += yl; }
  }
  if (lane == 31) { wtot[0][w] = xk; wtot[1][w] = xl; }
  __syncthreads();
  int bk = 0, bl = 0;
  for (int i = 0; i < w; ++i) { bk += wtot[0][i]; bl += wtot[1][i]; }
  if (tid < B) {
    s_vcu[tid + 1] = bk + xk;
    s_cu[tid + 1] = bl + xl;
  }
  if (tid == 0) { s_vcu[0] = 0; s_cu[0] = 0; }
  __syncthreads();
  if (blockIdx.x == 0) {
    for (int i = tid; i <= B; i += NT) {
      cu[i] = s_cu[i];
      if (vis_cu) vis_cu[i] = s_vcu[i];
    }
  }
  const int T = min(s_cu[B], T_cap);
  const int nv16 = W_vis / 8, nt16 = W_txt / 8;

  for (int r = blockIdx.x * (NT / 32) + w; r < T; r += gridDim.x * (NT / 32)) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (s_cu[mid] <= r) lo = mid; else hi = mid - 1;
    }
    const int b = lo;
    const int local = r - s_cu[b];
    if (lane == 0) pos[r] = local;
    const uint4* src;
    uint4* dst;
    int n16;
    if (local < s_cnt[b]) {
      const int j = __ldg(idx + (size_t)b * k_cap + local);
      const int n_img = bd.vis_off[b + 1] - bd.vis_off[b];
      if (j < 0 || j >= n_img) {
        if (lane == 0) set_error(err, SP_DEVERR_INDEX);
        continue;
      }
      src = reinterpret_cast<const uint4*>(X + (size_t)(bd.vis_off[b] + j) * W_vis);
      n16 = nv16;
      if (vis_packed) {
        const int vr = s_vcu[b] + local;
        if (lane == 0) vis_row_map[vr] = r;
        dst = reinterpret_cast<uint4*>(vis_packed + (size_t)vr * W_vis);
      } else {
        dst = reinterpret_cast<uint4*>(packed + (size_t)r * W_txt);
      }
    } else {
      src = reinterpret_cast<const uint4*>(text + (size_t)(bd.txt_off[b] + local - s_cnt[b]) * W_txt);
      dst = reinterpret_cast<uint4*>(packed + (size_t)r * W_txt);
      n16 = nt16;
    }
    copy_row(src, dst, n16, lane);
  }
}

}  // namespace

cudaError_t compact_launch(const BatchDesc& bd, const void* X, int W_vis, const void* text, int W_txt,
                           const int* idx, int k_cap, const int* count, void* packed, int* cu,
                           int* pos, void* vis_packed, int* vis_row_map, int* vis_cu, int T_cap,
                           int* err, cudaStream_t st) {
  const int rows_per_block = NT / 32;
  int grid = (T_cap + rows_per_block - 1) / rows_per_block;
  grid = std::max(1, std::min(grid, device_sm_count() * 8));
  prof_begin_launch(st);
  compact_kernel<<<grid, NT, 0, st>>>(bd, reinterpret_cast<const __nv_bfloat16*>(X), W_vis,
                                      reinterpret_cast<const __nv_bfloat16*>(text), W_txt, idx, k_cap,
                                      count, reinterpret_cast<__nv_bfloat16*>(packed), cu, pos,
                                      reinterpret_cast<__nv_bfloat16*>(vis_packed), vis_row_map, vis_cu,
                                      T_cap, err);
  prof_end_launch(st, SP_K_COMPACT, 0.0, 0.0);
  return cudaGetLastError();
}

}  // namespace sp
