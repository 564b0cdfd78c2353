// 3-D mRoPE of the Qwen2.5-VL backbone (Sec. 1) on the packed, pruned batch.
//
// mrope_positions_kernel writes each packed row's (t, h, w) rotary position:
// a kept visual token keeps its grid position in the unpruned image, the text
// after the image continues from the unpruned image block's largest position
// plus one (the reading of Sec. 3.3's last paragraph: the kept tokens stay in
// native order so the backbone's positional convention holds).
//
// mrope_rows_kernel turns those positions into one (cos, sin) row per packed
// row: pair i of the row takes the model's rotary table at the position
// component its section names.  The QKV GEMM's rotary epilogue then reads row r
// of this table at "position" r, so the GEMM itself is the same for 1-D RoPE and
// mRoPE; the gather is exact (the table itself is the model's fp64-computed one).
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

constexpr int MP_NT = 256;

__device__ __forceinline__ int warp_sum_int(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One CTA per image.
__global__ void __launch_bounds__(MP_NT)
mrope_positions_kernel(const BatchDesc bd, const GridDesc gd, const int* __restrict__ idx, int k_cap,
                       const int* __restrict__ count, int* __restrict__ pos3, int T_cap, int* err) {
  __shared__ int red[MP_NT / 32];
  const int b = blockIdx.x, tid = threadIdx.x;
  const int n_img = bd.vis_off[b + 1] - bd.vis_off[b];
  auto kept = [&](int c) {  // the image's kept count, as the compaction clamps it
    const int n = bd.vis_off[c + 1] - bd.vis_off[c];
    const int k = __ldg(count + c);
    return max(0, min(k, min(n, k_cap)));
  };
  // packed offset of this image: its predecessors' kept + text rows
  int part = 0;
  for (int c = tid; c < b; c += MP_NT) part += kept(c);
  part = warp_sum_int(part);
  if ((tid & 31) == 0) red[tid >> 5] = part;
  __syncthreads();
  int off = bd.txt_off[b];
  for (int w = 0; w < MP_NT / 32; ++w) off += red[w];
  const int k0 = __ldg(count + b);
  if (tid == 0 && (k0 < 0 || k0 > n_img || k0 > k_cap)) set_error(err, SP_DEVERR_INDEX);
  const int K = kept(b);
  const int L = bd.txt_off[b + 1] - bd.txt_off[b];
  const int gw = gd.grid_w[b];
  const int gh = (n_img + gw - 1) / gw;
  const int start = max(gh, gw);
  for (int j = tid; j < K + L; j += MP_NT) {
    const int r = off + j;
    if (r >= T_cap) {
      set_error(err, SP_DEVERR_INDEX);
      continue;
    }
    int4 p;
    if (j < K) {
      const int i = __ldg(idx + (size_t)b * k_cap + j);
      if (i < 0 || i >= n_img) {
        set_error(err, SP_DEVERR_INDEX);
        continue;
      }
      p = make_int4(0, i / gw, i % gw, 0);
    } else {
      const int q = start + (j - K);
      p = make_int4(q, q, q, 0);
    }
    reinterpret_cast<int4*>(pos3)[r] = p;
  }
}

// One warp per packed row; rows >= T only get their identity position.
__global__ void __launch_bounds__(256)
mrope_rows_kernel(const float2* __restrict__ rope, int max_pos, int half, const int* __restrict__ pos3, int s1,
                  int s2, const int* __restrict__ T_dev, int T_cap, float2* __restrict__ rows,
                  int* __restrict__ ident, int* err) {
  const int T = min(__ldg(T_dev), T_cap);
  const int lane = threadIdx.x & 31;
  for (int r = blockIdx.x * 8 + (threadIdx.x >> 5); r < T_cap; r += gridDim.x * 8) {
    if (lane == 0) ident[r] = r;
    if (r >= T) continue;
    const int4 p = __ldg(reinterpret_cast<const int4*>(pos3) + r);
    for (int i = lane; i < half; i += 32) {
      int q = i < s1 ? p.x : (i < s2 ? p.y : p.z);
      if (q < 0 || q >= max_pos) {
        set_error(err, SP_DEVERR_INDEX);
        q = 0;
      }
      rows[(size_t)r * half + i] = __ldg(rope + (size_t)q * half + i);
    }
  }
}

}  // namespace

cudaError_t mrope_positions_launch(const BatchDesc& bd, const GridDesc& gd, const int* idx, int k_cap,
                                   const int* count, int* pos3, int T_cap, int* err, cudaStream_t st) {
  prof_begin_launch(st);
  mrope_positions_kernel<<<bd.B, MP_NT, 0, st>>>(bd, gd, idx, k_cap, count, pos3, T_cap, err);
  prof_end_launch(st, SP_K_MISC, 0.0, 0.0);
  return cudaGetLastError();
}

cudaError_t mrope_rows_launch(const float2* rope, int max_pos, int half, const int* pos3, int s1, int s2,
                              const int* T_dev, int T_cap, float2* rows, int* ident, int* err, cudaStream_t st) {
  if (T_cap <= 0) return cudaSuccess;
  const int grid = std::min((T_cap + 7) / 8, device_sm_count() * 8);
  prof_begin_launch(st);
  mrope_rows_kernel<<<grid, 256, 0, st>>>(rope, max_pos, half, pos3, s1, s2, T_dev, T_cap, rows, ident, err);
  prof_end_launch(st, SP_K_MISC, 0.0, (double)T_cap * half * 8.0);
  return cudaGetLastError();
}

}  // namespace sp
