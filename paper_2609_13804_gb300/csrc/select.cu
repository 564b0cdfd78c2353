// Sequential pointer selection (Sec. 3.2, Eq. 4; grouped rounds Sec. 3.5, Eq. 11;
// Algorithm 1 steps 2-4) as one persistent kernel per batch.
//
// One thread-block cluster of C CTAs runs one episode (an image, or one
// candidate group of it) for all of its rounds without leaving the GPU.  The
// candidates are split into C contiguous slices; each CTA keeps its slice of
// the folded pointer keys in shared memory for the whole episode.  A round:
//   1. attention of the last history position over the history: CTA c takes
//      positions c, c+C, ...; each warp loads all rows it needs for the round
//      at once (query, key and value rows of its positions) so the round pays
//      one L2 latency, and the warps' partials (max, sum, weighted values) are
//      folded into the CTA's partial;
//   2. cluster barrier; every CTA merges the C partials read over DSMEM in rank
//      order (so all CTAs hold bitwise-identical results), adds the residual and
//      applies LN2 -> pointer query;
//   3. every CTA scores its available candidates from shared memory and keeps
//      its top g+1 (logit desc, index asc); the raw STOP logit is computed by
//      every CTA identically;
//   4. cluster barrier; every CTA merges the C lists, takes the same decision
//      (STOP iff strictly above the best available visual logit, else TopG
//      truncated to the cap), masks its own slice and extends the history.
// The decoder matrices are folded on the host side of the ABI so that no
// matrix-vector product remains inside the loop:
//   QS = x Wq_s^T / sqrt(h), KS = x Wk_s^T, VT = x (Wo_s Wv_s)^T   (x = LN1(W_in m))
//   KT = m (Wq_p^T Wk_p)^T / sqrt(h),  so  l(j) = <LN2(u), KT_j>,
//   u = Z_last + sum_i softmax_i(<QS_last, KS_i>) VT_i.
// Double-buffered exchange slots make two cluster barriers per round enough.
#include <cooperative_groups.h>

#include <climits>

#include "common.cuh"
#include "internal.h"

namespace cg = cooperative_groups;

namespace sp {

namespace {

constexpr int NT = 256;
constexpr int NW = NT / 32;
constexpr int GMAX = 16;  // largest g; lists hold g + 1 entries

struct SelSmem {
  size_t kt, stopkt, wpart_o, wpart_ml, part_o, part_ml, top_v, top_i, u, xp, lg, taken, hist, misc, total;
};

__host__ __device__ inline size_t al16(size_t x) { return (x + 15) & ~size_t(15); }

__host__ __device__ inline SelSmem sel_layout(int h, int n_loc, int k_max, int C, bool keys_in_smem) {
  SelSmem L;
  size_t o = 0;
  (void)C;
  L.kt = o;       o += al16(keys_in_smem ? (size_t)n_loc * h * 4 : 0);
  L.stopkt = o;   o += al16((size_t)h * 4);
  L.wpart_o = o;  o += al16((size_t)NW * h * 4);
  L.wpart_ml = o; o += al16((size_t)NW * 2 * 4);
  L.part_o = o;   o += al16((size_t)2 * h * 4);
  L.part_ml = o;  o += al16(2 * 2 * 4);
  L.top_v = o;    o += al16(2 * (GMAX + 1) * 4);
  L.top_i = o;    o += al16(2 * (GMAX + 1) * 4);
  L.u = o;        o += al16((size_t)h * 4);
  L.xp = o;       o += al16((size_t)h * 4);
  L.lg = o;       o += al16((size_t)n_loc * 4);
  L.taken = o;    o += al16((size_t)n_loc);
  L.hist = o;     o += al16((size_t)(k_max + 1) * 4);
  L.misc = o;     o += al16(128 * 4);
  L.total = o;
  return L;
}

SP_DEVINL bool better(float v, int i, float bv, int bi) { return v > bv || (v == bv && i < bi); }

SP_DEVINL void warp_best(float& v, int& i) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, i, o);
    if (better(ov, oi, v, i)) { v = ov; i = oi; }
  }
}

SP_DEVINL float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = (l < NW) ? red[l] : 0.f;
  return warp_sum(t);
}

SP_DEVINL float dot4(const float4& a, const float4& b) { return a.x * b.x + a.y * b.y + a.z * b.z + a.w * b.w; }

// HV = h / 128: float4 slices per lane of an h-vector (lane holds elements
// 4 (lane + 32 k) .. +3, k < HV).  P = history positions a warp loads at once.
template <int HV>
__global__ void __launch_bounds__(NT, 1)
select_kernel(const BatchDesc bd, const SelectArgs a, int n_loc_max, int keys_in_smem) {
  constexpr int P = (16 / HV) > 0 ? 16 / HV : 1;
  constexpr int DPT = (HV * 128) / NT > 0 ? (HV * 128) / NT : 1;  // dims per thread in the merges
  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int rank = (int)cluster.block_rank();
  const int e = blockIdx.x / C;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int h = a.h, k_max = a.k_max, g = a.g;

  // episode geometry
  int lo = 0, hi = bd.B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (bd.ep_off[mid] <= e) lo = mid; else hi = mid - 1;
  }
  const int b = lo;
  const int n_img = bd.vis_off[b + 1] - bd.vis_off[b];
  const int gs = bd.group_size > 0 ? bd.group_size : n_img;
  const int c0 = (e - bd.ep_off[b]) * gs;
  const int n_e = min(gs, n_img - c0);
  const int row0 = bd.vis_off[b] + c0;
  const int n_loc = (n_e + C - 1) / C;
  const int j0 = rank * n_loc;
  const int nl = max(0, min(j0 + n_loc, n_e) - j0);

  extern __shared__ __align__(16) uint8_t sm[];
  const SelSmem L = sel_layout(h, n_loc_max, k_max, C, keys_in_smem != 0);
  float* kt_s = reinterpret_cast<float*>(sm + L.kt);
  float* stopkt = reinterpret_cast<float*>(sm + L.stopkt);
  float* wpart_o = reinterpret_cast<float*>(sm + L.wpart_o);
  float* wpart_ml = reinterpret_cast<float*>(sm + L.wpart_ml);
  float* part_o = reinterpret_cast<float*>(sm + L.part_o);
  float* part_ml = reinterpret_cast<float*>(sm + L.part_ml);
  float* top_v = reinterpret_cast<float*>(sm + L.top_v);
  int* top_i = reinterpret_cast<int*>(sm + L.top_i);
  float* u_s = reinterpret_cast<float*>(sm + L.u);
  float* xp_s = reinterpret_cast<float*>(sm + L.xp);
  float* lg = reinterpret_cast<float*>(sm + L.lg);
  uint8_t* taken = sm + L.taken;
  int* hist = reinterpret_cast<int*>(sm + L.hist);
  float* misc = reinterpret_cast<float*>(sm + L.misc);
  float* red = misc;                                  // [0, 32)
  float* rm = misc + 32;                              // [32, 48)  peer maxima
  float* rl = misc + 48;                              // [48, 64)  peer sums
  float* gtop_v = misc + 64;                          // [64, 81)
  int* gtop_i = reinterpret_cast<int*>(misc + 96);    // [96, 113)

  // stage this CTA's slice of the folded keys and the STOP key
  const float* KT = a.KT;
  const int h4 = h >> 2;
  if (keys_in_smem) {
    for (int i = tid; i < nl * h4; i += NT) {
      const int j = i / h4, c = i % h4;
      reinterpret_cast<float4*>(kt_s)[(size_t)j * h4 + c] =
          __ldg(reinterpret_cast<const float4*>(KT + (size_t)(row0 + j0 + j) * a.ldkt) + c);
    }
  }
  for (int i = tid; i < h4; i += NT)
    reinterpret_cast<float4*>(stopkt)[i] = __ldg(reinterpret_cast<const float4*>(KT + (size_t)a.stop_row * a.ldkt) + i);
  for (int j = tid; j < n_loc_max; j += NT) taken[j] = 0;
  if (tid == 0) hist[0] = a.start_row;
  const float bias = __ldg(a.stop_bias + e);
  const size_t trace = (size_t)e * (k_max + 1);
  __syncthreads();

  int nsel = 0, round = 0;
  while (nsel < k_max) {
    const int n_avail = n_e - nsel;
    if (n_avail == 0) {  // only STOP remains: it wins this round
      if (rank == 0 && tid == 0) {
        if (a.margin) a.margin[trace + round] = INFINITY;
        if (a.gap) a.gap[trace + round] = -INFINITY;
      }
      ++round;
      break;
    }
    const int buf = round & 1;
    const int t = nsel + 1;
    const int last = hist[t - 1];

    // ---- 1. partial causal self-attention of the last position.  Every load
    //      of the round (query, residual, owned history rows) is issued at once.
    float zr[DPT];
#pragma unroll
    for (int d = 0; d < DPT; ++d) zr[d] = (tid + d * NT < h) ? __ldg(a.Z + (size_t)last * a.ldz + tid + d * NT) : 0.f;
    float4 q[HV];
    const float4* qrow = reinterpret_cast<const float4*>(a.QS + (size_t)last * a.ldqs);
#pragma unroll
    for (int k = 0; k < HV; ++k) q[k] = __ldg(qrow + lane + 32 * k);
    const int np = (rank < t) ? (t - 1 - rank) / C + 1 : 0;  // positions rank, rank + C, ...
    float m_w = -INFINITY, l_w = 0.f;
    float4 o_w[HV];
#pragma unroll
    for (int k = 0; k < HV; ++k) o_w[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int k0 = warp * P; k0 < np; k0 += NW * P) {
      float4 kr[P][HV], vr[P][HV];
#pragma unroll
      for (int pp = 0; pp < P; ++pp) {
        if (k0 + pp < np) {
          const int row = hist[rank + (k0 + pp) * C];
          const float4* ks = reinterpret_cast<const float4*>(a.KS + (size_t)row * a.ldks);
          const float4* vt = reinterpret_cast<const float4*>(a.VT + (size_t)row * a.ldvt);
#pragma unroll
          for (int k = 0; k < HV; ++k) {
            kr[pp][k] = __ldg(ks + lane + 32 * k);
            vr[pp][k] = __ldg(vt + lane + 32 * k);
          }
        }
      }
#pragma unroll
      for (int pp = 0; pp < P; ++pp) {
        if (k0 + pp < np) {
          float s = 0.f;
#pragma unroll
          for (int k = 0; k < HV; ++k) s += dot4(q[k], kr[pp][k]);
          s = warp_sum(s);
          const float mn = fmaxf(m_w, s);
          const float cw = (m_w == -INFINITY) ? 0.f : expf(m_w - mn);
          const float ps = expf(s - mn);
          l_w = l_w * cw + ps;
#pragma unroll
          for (int k = 0; k < HV; ++k) {
            o_w[k].x = o_w[k].x * cw + ps * vr[pp][k].x;
            o_w[k].y = o_w[k].y * cw + ps * vr[pp][k].y;
            o_w[k].z = o_w[k].z * cw + ps * vr[pp][k].z;
            o_w[k].w = o_w[k].w * cw + ps * vr[pp][k].w;
          }
          m_w = mn;
        }
      }
    }
#pragma unroll
    for (int k = 0; k < HV; ++k) reinterpret_cast<float4*>(wpart_o + warp * h)[lane + 32 * k] = o_w[k];
    if (lane == 0) {
      wpart_ml[warp * 2 + 0] = m_w;
      wpart_ml[warp * 2 + 1] = l_w;
    }
    __syncthreads();
    {  // this CTA's partial from its warps' partials (warp order)
      float m_c = -INFINITY;
#pragma unroll
      for (int w = 0; w < NW; ++w) m_c = fmaxf(m_c, wpart_ml[w * 2]);
      float cw[NW];
      float l_c = 0.f;
#pragma unroll
      for (int w = 0; w < NW; ++w) {
        const float mw = wpart_ml[w * 2];
        cw[w] = (mw == -INFINITY) ? 0.f : expf(mw - m_c);
        l_c += cw[w] * wpart_ml[w * 2 + 1];
      }
      float* po = part_o + buf * h;
#pragma unroll
      for (int d = 0; d < DPT; ++d) {
        const int i = tid + d * NT;
        if (i >= h) continue;
        float acc = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) acc += cw[w] * wpart_o[w * h + i];
        po[i] = acc;
      }
      if (tid == 0) {
        part_ml[buf * 2 + 0] = m_c;
        part_ml[buf * 2 + 1] = l_c;
      }
    }
    cluster.sync();

    // ---- 2. merge partials (rank order), residual, LN2
    if (tid < C) {
      const float* pm = cluster.map_shared_rank(part_ml, tid);
      rm[tid] = pm[buf * 2 + 0];
      rl[tid] = pm[buf * 2 + 1];
    }
    __syncthreads();
    float m = -INFINITY;
    for (int r = 0; r < C; ++r) m = fmaxf(m, rm[r]);
    float wsum = 0.f;
    float wr[16];
#pragma unroll
    for (int r = 0; r < 16; ++r) {
      wr[r] = 0.f;
      if (r < C && rm[r] != -INFINITY) wr[r] = expf(rm[r] - m);
      if (r < C) wsum += wr[r] * rl[r];
    }
    const float inv = 1.f / wsum;
    float s_loc = 0.f;
    float uv[DPT];
#pragma unroll
    for (int d = 0; d < DPT; ++d) {
      const int i = tid + d * NT;
      uv[d] = 0.f;
      if (i >= h) continue;
      float ro[16];
#pragma unroll
      for (int r = 0; r < 16; ++r) ro[r] = (r < C) ? cluster.map_shared_rank(part_o, r)[buf * h + i] : 0.f;
      float o = 0.f;
#pragma unroll
      for (int r = 0; r < 16; ++r) o += wr[r] * ro[r];
      uv[d] = zr[d] + o * inv;
      s_loc += uv[d];
    }
    const float mean = block_sum(s_loc, red) / (float)h;
    float v_loc = 0.f;
#pragma unroll
    for (int d = 0; d < DPT; ++d) {
      const float c = (tid + d * NT < h) ? uv[d] - mean : 0.f;
      v_loc += c * c;
    }
    const float rstd = rsqrtf(block_sum(v_loc, red) / (float)h + a.ln_eps);
#pragma unroll
    for (int d = 0; d < DPT; ++d) {
      const int i = tid + d * NT;
      if (i >= h) continue;
      float x = (uv[d] - mean) * rstd;
      if (a.ln2_g) x *= __ldg(a.ln2_g + i);
      if (a.ln2_b) x += __ldg(a.ln2_b + i);
      xp_s[i] = x;
    }
    __syncthreads();

    // ---- 3. logits of the available local candidates and the raw STOP logit
    float4 xr[HV];
#pragma unroll
    for (int k = 0; k < HV; ++k) xr[k] = reinterpret_cast<const float4*>(xp_s)[lane + 32 * k];
    for (int j = warp; j < nl; j += NW) {
      if (taken[j]) {
        if (lane == 0) lg[j] = -INFINITY;
        continue;
      }
      const float4* kr = keys_in_smem ? reinterpret_cast<const float4*>(kt_s + (size_t)j * h)
                                      : reinterpret_cast<const float4*>(KT + (size_t)(row0 + j0 + j) * a.ldkt);
      float s = 0.f;
#pragma unroll
      for (int k = 0; k < HV; ++k) s += dot4(xr[k], kr[lane + 32 * k]);
      s = warp_sum(s);
      if (lane == 0) lg[j] = s;
    }
    float stop_raw = 0.f;
    {
      float s = 0.f;
#pragma unroll
      for (int k = 0; k < HV; ++k) s += dot4(xr[k], reinterpret_cast<const float4*>(stopkt)[lane + 32 * k]);
      stop_raw = warp_sum(s);  // every warp of every CTA computes the same value
    }
    __syncthreads();

    // local top g+1 by (logit desc, index asc)
    if (warp == 0) {
      int picked[GMAX + 1];
      for (int r = 0; r <= g; ++r) {
        float bv = -INFINITY;
        int bi = INT_MAX;
        for (int j = lane; j < nl; j += 32) {
          const float v = lg[j];
          if (v == -INFINITY) continue;
          bool ex = false;
          for (int q2 = 0; q2 < r; ++q2) ex |= (picked[q2] == j);
          if (!ex && better(v, j, bv, bi)) { bv = v; bi = j; }
        }
        warp_best(bv, bi);
        picked[r] = bi;
        if (lane == 0) {
          top_v[buf * (GMAX + 1) + r] = bv;
          top_i[buf * (GMAX + 1) + r] = (bi == INT_MAX) ? INT_MAX : j0 + bi;
        }
      }
    }
    cluster.sync();

    // ---- 4. merge the C lists (identically in every CTA) and decide
    if (warp == 0) {
      const int per = g + 1;
      const int tot = C * per;
      float ev[9];
      int ei[9];
#pragma unroll
      for (int k = 0; k < 9; ++k) {
        const int idx = lane + 32 * k;
        ev[k] = -INFINITY;
        ei[k] = INT_MAX;
        if (idx < tot) {
          const int r = idx / per, s2 = idx % per;
          const float* rv = cluster.map_shared_rank(top_v, r);
          const int* ri = cluster.map_shared_rank(top_i, r);
          ev[k] = rv[buf * (GMAX + 1) + s2];
          ei[k] = ri[buf * (GMAX + 1) + s2];
          if (ei[k] == INT_MAX) ev[k] = -INFINITY;
        }
      }
      for (int r = 0; r < per; ++r) {
        float bv = -INFINITY;
        int bi = INT_MAX;
#pragma unroll
        for (int k = 0; k < 9; ++k)
          if (better(ev[k], ei[k], bv, bi)) { bv = ev[k]; bi = ei[k]; }
        warp_best(bv, bi);
#pragma unroll
        for (int k = 0; k < 9; ++k)
          if (ei[k] == bi) { ev[k] = -INFINITY; ei[k] = INT_MAX; }
        if (lane == 0) {
          gtop_v[r] = bv;
          gtop_i[r] = bi;
        }
      }
    }
    __syncthreads();
    const float stop_logit = stop_raw + bias;
    const float best = gtop_v[0];
    if (rank == 0 && tid == 0) {
      if (a.gap) a.gap[trace + round] = best - stop_raw;
      if (a.margin) {
        // smallest gap between consecutive values among the top g+1 of
        // {available visual logits} U {STOP}
        float vals[GMAX + 2];
        int n = 0;
        const int nv = min(g + 1, n_avail);
        for (int k = 0; k < nv; ++k) vals[n++] = gtop_v[k];
        int ins = n;
        while (ins > 0 && vals[ins - 1] < stop_logit) --ins;
        for (int k = n; k > ins; --k) vals[k] = vals[k - 1];
        vals[ins] = stop_logit;
        ++n;
        const int use = min(n, g + 1);
        float mg = INFINITY;
        for (int k = 0; k + 1 < use; ++k) mg = fminf(mg, vals[k] - vals[k + 1]);
        a.margin[trace + round] = mg;
      }
    }
    ++round;
    if (stop_logit > best) break;  // STOP
    const int take = min(min(g, k_max - nsel), n_avail);
    if (tid == 0) {
      for (int k = 0; k < take; ++k) {
        const int jj = gtop_i[k];
        if (jj < 0 || jj >= n_e) {
          set_error(a.err, SP_DEVERR_INDEX);
          hist[t + k] = a.start_row;
          continue;
        }
        hist[t + k] = row0 + jj;
        if (jj >= j0 && jj < j0 + nl) taken[jj - j0] = 1;
        if (rank == 0 && a.order) a.order[(size_t)e * k_max + nsel + k] = jj;
      }
    }
    nsel += take;
    __syncthreads();
  }
  if (rank == 0 && tid == 0) {
    if (a.ep_count) a.ep_count[e] = nsel;
    if (a.rounds) a.rounds[e] = round;
  }
  cluster.sync();  // peers may still read this CTA's slots
}

// Algorithm 1 step 4: per image, the union of its episodes' selections in
// native (ascending) order, -1 padded to k_cap.
__global__ void __launch_bounds__(512)
restore_kernel(const BatchDesc bd, const int* __restrict__ order, const int* __restrict__ ep_count,
               int k_max, int* __restrict__ idx, int k_cap, int* __restrict__ count, int* err) {
  extern __shared__ uint8_t flags[];
  __shared__ int wsum[32];
  const int b = blockIdx.x, tid = threadIdx.x, NTR = blockDim.x;
  const int n_img = bd.vis_off[b + 1] - bd.vis_off[b];
  const int gs = bd.group_size > 0 ? bd.group_size : n_img;
  for (int i = tid; i < n_img; i += NTR) flags[i] = 0;
  __syncthreads();
  for (int e = bd.ep_off[b]; e < bd.ep_off[b + 1]; ++e) {
    const int c0 = (e - bd.ep_off[b]) * gs;
    const int cnt = ep_count[e];
    for (int i = tid; i < cnt; i += NTR) {
      const int j = order[(size_t)e * k_max + i];
      if (j < 0 || c0 + j >= n_img || j >= gs) { set_error(err, SP_DEVERR_INDEX); continue; }
      flags[c0 + j] = 1;
    }
  }
  __syncthreads();
  const int chunk = (n_img + NTR - 1) / NTR;
  const int s = tid * chunk, en = min(s + chunk, n_img);
  int c = 0;
  for (int i = s; i < en; ++i) c += flags[i];
  // exclusive block scan of c
  const int lane = tid & 31, w = tid >> 5;
  int x = c;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[w] = x;
  __syncthreads();
  if (w == 0) {
    int v = (lane < (NTR >> 5)) ? wsum[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, v, o);
      if (lane >= o) v += y;
    }
    wsum[lane] = v;
  }
  __syncthreads();
  const int total = wsum[(NTR >> 5) - 1];
  int off = x - c + (w > 0 ? wsum[w - 1] : 0);
  int* row = idx + (size_t)b * k_cap;
  for (int i = s; i < en; ++i) {
    if (flags[i]) {
      if (off < k_cap) row[off] = i;
      ++off;
    }
  }
  for (int i = total + tid; i < k_cap; i += NTR) row[i] = -1;
  if (tid == 0) {
    if (total > k_cap) set_error(err, SP_DEVERR_INDEX);
    count[b] = min(total, k_cap);
  }
}

}  // namespace

int select_cluster_size(const BatchDesc& bd, int h, bool* keys_in_smem, size_t* smem_bytes) {
  int n_max = 0;
  for (int b = 0; b < bd.B; ++b) {
    const int n = bd.vis_off[b + 1] - bd.vis_off[b];
    n_max = std::max(n_max, bd.group_size > 0 ? std::min(bd.group_size, n) : n);
  }
  (void)smem_bytes;
  const size_t budget = 200 * 1024;
  for (int C : {8, 16}) {
    const int n_loc = (n_max + C - 1) / C;
    if ((size_t)n_loc * h * 4 + 16 * 1024 <= budget) {
      *keys_in_smem = true;
      return C;
    }
  }
  *keys_in_smem = false;
  return 16;
}

cudaError_t select_launch(const BatchDesc& bd, int n_episodes, const SelectArgs& a, int C,
                          bool keys_in_smem, size_t /*unused*/, cudaStream_t st) {
  if (n_episodes <= 0) return cudaSuccess;
  int n_max = 0;
  for (int b = 0; b < bd.B; ++b) {
    const int n = bd.vis_off[b + 1] - bd.vis_off[b];
    n_max = std::max(n_max, bd.group_size > 0 ? std::min(bd.group_size, n) : n);
  }
  const int n_loc = (n_max + C - 1) / C;
  const SelSmem L = sel_layout(a.h, n_loc, a.k_max, C, keys_in_smem);
  void (*kern)(const BatchDesc, const SelectArgs, int, int) = nullptr;
  switch (a.h / 128) {
    case 1: kern = select_kernel<1>; break;
    case 2: kern = select_kernel<2>; break;
    case 4: kern = select_kernel<4>; break;
    case 8: kern = select_kernel<8>; break;
    default: return cudaErrorInvalidValue;
  }
  cudaError_t r = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L.total);
  if (r != cudaSuccess) return r;
  if (C > 8) {
    r = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (r != cudaSuccess) return r;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_episodes * C, 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = L.total;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  prof_begin_launch(st);
  r = cudaLaunchKernelEx(&cfg, kern, bd, a, n_loc, keys_in_smem ? 1 : 0);
  prof_end_launch(st, SP_K_SELECT, 0.0, 0.0);
  return r;
}

cudaError_t restore_launch(const BatchDesc& bd, const int* order, const int* ep_count, int k_max,
                           int* idx, int k_cap, int* count, int* err, cudaStream_t st) {
  int n_max = 1;
  for (int b = 0; b < bd.B; ++b) n_max = std::max(n_max, bd.vis_off[b + 1] - bd.vis_off[b]);
  if (n_max > 48 * 1024) {
    cudaError_t r = cudaFuncSetAttribute(restore_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, n_max);
    if (r != cudaSuccess) return r;
  }
  prof_begin_launch(st);
  restore_kernel<<<bd.B, 512, n_max, st>>>(bd, order, ep_count, k_max, idx, k_cap, count, err);
  prof_end_launch(st, SP_K_RESTORE, 0.0, 0.0);
  return cudaGetLastError();
}

}  // namespace sp
