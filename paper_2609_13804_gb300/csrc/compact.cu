// Compaction (Algorithm 1 step 5, X_S = Gather(X, S)): the kept visual rows of
// every image, in native order, followed by its text rows, written as one packed
// variable-length buffer with cu_seqlens and per-sequence positions.  Pure data
// movement, HBM-bound: rows are cut into 2 KB pieces and a warp moves three
// pieces per pass with 16-byte vector copies.
//
// Every block recomputes the (small) prefix sums of the per-image counts from
// the device counts, so the kernel needs no host round trip and no second
// launch; block 0 publishes cu_seqlens / vis_cu.
//
// Index mode (vis_src): the kept visual rows are not copied; the kernel writes,
// for each, the row of X it comes from (with vis_row_map, its packed row), and
// the projector's first GEMM gathers those rows from X as its operand.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

constexpr int NT = 256;

__global__ void __launch_bounds__(NT, 2)
compact_kernel(const BatchDesc bd, const __nv_bfloat16* __restrict__ X, int W_vis,
               const __nv_bfloat16* __restrict__ text, int W_txt, const int* __restrict__ idx, int k_cap,
               const int* __restrict__ count, __nv_bfloat16* __restrict__ packed, int* __restrict__ cu,
               int* __restrict__ pos, __nv_bfloat16* __restrict__ vis_packed, int* __restrict__ vis_row_map,
               int* __restrict__ vis_cu, int* __restrict__ vis_src, int T_cap, int* err) {
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
  const int gw = blockIdx.x * (NT / 32) + w, nw = gridDim.x * (NT / 32);
  // The copy is cut into pieces of at most PIECE16 16-byte chunks (2 KB): a
  // visual row of 1,024 bf16 is one piece, a text row of 4,096 bf16 four.
  // Visual pieces come first, then text pieces.  A warp takes PPW pieces per
  // pass: it locates their rows (the visual rows' index loads go out
  // together), then loads every chunk of the PPW pieces before storing any
  // (12 loads per lane, 6 KB per warp in flight).
  constexpr int PPW = 3, PIECE16 = 128;
  const int V = s_vcu[B], Lt = bd.txt_off[B];
  const int ppv = vis_src ? 1 : (nv16 + PIECE16 - 1) / PIECE16, ppt = (nt16 + PIECE16 - 1) / PIECE16;
  const int NPv = V * ppv, NP = NPv + Lt * ppt;
  for (int p0 = gw * PPW; p0 < NP; p0 += nw * PPW) {
    const uint4* src[PPW];
    uint4* dst[PPW];
    int nc[PPW], jv[PPW], vb[PPW], c0v[PPW], vrv[PPW];
#pragma unroll
    for (int u = 0; u < PPW; ++u) {
      const int pc = p0 + u;
      nc[u] = 0;
      jv[u] = -1;
      vb[u] = -1;
      c0v[u] = 0;
      vrv[u] = -1;
      src[u] = nullptr;
      dst[u] = nullptr;
      if (pc >= NP) continue;
      if (pc < NPv) {  // a piece of kept visual row vr
        const int vr = pc / ppv, sub = pc - vr * ppv;
        int lo = 0, hi = B - 1;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (s_vcu[mid] <= vr) lo = mid; else hi = mid - 1;
        }
        const int local = vr - s_vcu[lo];
        const int r = s_cu[lo] + local;
        if (r >= T) continue;
        jv[u] = __ldg(idx + (size_t)lo * k_cap + local);  // resolved below, with every index load out
        vb[u] = lo;
        vrv[u] = vr;
        const int c0 = sub * PIECE16;
        c0v[u] = c0;
        nc[u] = vis_src ? 0 : min(PIECE16, nv16 - c0);
        dst[u] = (vis_packed ? reinterpret_cast<uint4*>(vis_packed + (size_t)vr * W_vis)
                             : reinterpret_cast<uint4*>(packed + (size_t)r * W_txt)) + c0;
        if (sub == 0 && lane == 0) {
          pos[r] = local;
          if (vis_packed || vis_src) vis_row_map[vr] = r;
        }
      } else {  // a piece of text row tr
        const int tp = pc - NPv;
        const int tr = tp / ppt, sub = tp - tr * ppt;
        int lo = 0, hi = B - 1;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (bd.txt_off[mid] <= tr) lo = mid; else hi = mid - 1;
        }
        const int local = s_cnt[lo] + (tr - bd.txt_off[lo]);
        const int r = s_cu[lo] + local;
        if (r >= T) continue;
        const int c0 = sub * PIECE16;
        nc[u] = min(PIECE16, nt16 - c0);
        src[u] = reinterpret_cast<const uint4*>(text + (size_t)tr * W_txt) + c0;
        dst[u] = reinterpret_cast<uint4*>(packed + (size_t)r * W_txt) + c0;
        if (sub == 0 && lane == 0) pos[r] = local;
      }
    }
#pragma unroll
    for (int u = 0; u < PPW; ++u) {
      if (vb[u] < 0) continue;
      const int n_img = bd.vis_off[vb[u] + 1] - bd.vis_off[vb[u]];
      if (jv[u] < 0 || jv[u] >= n_img) {
        if (lane == 0) {
          set_error(err, SP_DEVERR_INDEX);
          if (vis_src) vis_src[vrv[u]] = -1;  // (a gather of row -1 reads zeros)
        }
        nc[u] = 0;
        continue;
      }
      src[u] = reinterpret_cast<const uint4*>(X + (size_t)(bd.vis_off[vb[u]] + jv[u]) * W_vis) + c0v[u];
      if (vis_src && lane == 0) vis_src[vrv[u]] = bd.vis_off[vb[u]] + jv[u];
    }
    uint4 x[PPW][PIECE16 / 32];
#pragma unroll
    for (int u = 0; u < PPW; ++u)
#pragma unroll
      for (int q = 0; q < PIECE16 / 32; ++q)
        if (lane + q * 32 < nc[u]) x[u][q] = __ldg(src[u] + lane + q * 32);
#pragma unroll
    for (int u = 0; u < PPW; ++u)
#pragma unroll
      for (int q = 0; q < PIECE16 / 32; ++q)
        if (lane + q * 32 < nc[u]) dst[u][lane + q * 32] = x[u][q];
  }
}

}  // namespace

cudaError_t compact_launch(const BatchDesc& bd, const void* X, int W_vis, const void* text, int W_txt,
                           const int* idx, int k_cap, const int* count, void* packed, int* cu,
                           int* pos, void* vis_packed, int* vis_row_map, int* vis_cu, int* vis_src, int T_cap,
                           int* err, cudaStream_t st) {
  // pieces of at most 2 KB (one per visual row of 1,024 bf16, more for wider
  // rows), three per warp and pass
  const long long pieces = (long long)T_cap * ((std::max(W_vis, W_txt) / 8 + 127) / 128);
  int grid = (int)std::min<long long>((pieces + NT / 32 * 3 - 1) / (NT / 32 * 3), 1 << 20);
  grid = std::max(1, std::min(grid, device_sm_count() * 2));  // resident: two CTAs per SM
  prof_begin_launch(st);
  compact_kernel<<<grid, NT, 0, st>>>(bd, reinterpret_cast<const __nv_bfloat16*>(X), W_vis,
                                      reinterpret_cast<const __nv_bfloat16*>(text), W_txt, idx, k_cap,
                                      count, reinterpret_cast<__nv_bfloat16*>(packed), cu, pos,
                                      reinterpret_cast<__nv_bfloat16*>(vis_packed), vis_row_map, vis_cu,
                                      vis_src, T_cap, err);
  prof_end_launch(st, SP_K_COMPACT, 0.0, 0.0);
  return cudaGetLastError();
}

}  // namespace sp
