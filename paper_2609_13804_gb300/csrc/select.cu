// Sequential pointer selection (Sec. 3.2, Eq. 4; grouped rounds Sec. 3.5, Eq. 11;
// Algorithm 1 steps 2-4) as one persistent kernel per batch.
//
// One thread-block cluster of C CTAs runs one episode (an image, or one
// candidate group of it) for all of its rounds without leaving the GPU.  The
// candidates are split into C contiguous slices; each CTA keeps its slice of
// the folded pointer keys in shared memory for the whole episode.  A round:
//   1. attention of the last history position over the history: CTA c takes
//      positions c, c+C, ...; each warp loads all rows it needs for the round
//      at once (query, key and value rows of its positions), the warps'
//      partials (max, sum, weighted values) fold into the CTA's partial, which
//      the CTA pushes into its slot in every CTA's shared memory;
//   2. cluster barrier; every CTA merges the C partials from its own shared
//      memory in rank order (so all CTAs hold bitwise-identical results), adds
//      the residual and applies LN2 -> pointer query;
//   3. every CTA scores its available candidates from shared memory (four per
//      warp iteration, shuffle reductions interleaved), each warp keeping a
//      running top g+1 (logit desc, index asc); warp 0 merges them and pushes
//      the CTA's list into every CTA; the raw STOP logit is computed by every
//      CTA identically;
//   4. cluster barrier; every CTA merges the C lists, takes the same decision
//      (STOP iff strictly above the best available visual logit, else TopG
//      truncated to the cap), masks its own slice and extends the history.
// Exchanges are pushes (remote stores before the barrier, local loads after),
// double-buffered by round parity, so two cluster barriers per round suffice.
// The decoder matrices are folded on the host side of the ABI so that no
// matrix-vector product remains inside the loop:
//   QS = x Wq_s^T / sqrt(h), KS = x Wk_s^T, VT = x (Wo_s Wv_s)^T   (x = LN1(W_in m))
//   KT = m (Wq_p^T Wk_p)^T / sqrt(h),  so  l(j) = <LN2(u), KT_j>,
//   u = Z_last + sum_i softmax_i(<QS_last, KS_i>) VT_i.
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
  size_t kt, lgp, stopkt, wpart_o, wpart_ml, all_o, all_ml, wtop_v, wtop_i, all_tv, all_ti, xp, taken, hist, misc,
      wsm, all_sm, score, mx, ma, mc, mn, v3, hb, xo, total;
};

__host__ __device__ inline size_t al16(size_t x) { return (x + 15) & ~size_t(15); }

// Shared-memory layout.  The all_* slots receive, per round parity, one entry
// per CTA of the cluster, written remotely by that CTA (push exchange).
__host__ __device__ inline SelSmem sel_layout(int h, int n_loc, int k_max, int C, bool keys_in_smem,
                                              bool multi = false) {
  SelSmem L;
  size_t o = 0;
  // keys in shared memory: dims-major, (n_loc + 1) columns (the last one is
  // STOP's key), float4 (d4, j) at d4 * (n_loc + 1) + j
  L.kt = o;       o += al16(keys_in_smem ? (size_t)(n_loc + 1) * h * 4 : 0);
  L.lgp = o;      o += al16(keys_in_smem ? (size_t)NW * (n_loc + 1) * 4 : 0);
  L.stopkt = o;   o += al16((size_t)h * 4);
  L.wpart_o = o;  o += al16((size_t)NW * h * 4);
  L.wpart_ml = o; o += al16((size_t)NW * 2 * 4);
  L.all_o = o;    o += al16((size_t)2 * C * h * 4);
  L.all_ml = o;   o += al16((size_t)2 * C * 2 * 4);
  L.wtop_v = o;   o += al16((size_t)NW * (GMAX + 1) * 4);
  L.wtop_i = o;   o += al16((size_t)NW * (GMAX + 1) * 4);
  L.all_tv = o;   o += al16((size_t)2 * C * (GMAX + 1) * 4);
  L.all_ti = o;   o += al16((size_t)2 * C * (GMAX + 1) * 4);
  L.xp = o;       o += al16((size_t)h * 4);
  L.taken = o;    o += al16((size_t)n_loc);
  L.hist = o;     o += al16((size_t)(k_max + 1) * 4);
  L.misc = o;     o += al16(128 * 4);
  // training pathway: per-warp / per-CTA softmax partials (max, sum) and the
  // CTA's scores of Eq. 6
  L.wsm = o;      o += al16((size_t)NW * 2 * 4);
  L.all_sm = o;   o += al16((size_t)2 * C * 2 * 4);
  L.score = o;    o += al16((size_t)n_loc * 4);
  // decoders of several layers: the new position's residual, its running
  // attention / cross-attention output (updated in place), a normalised input
  // (h each), and the pushed matrix-vector products.  Aliases: the pushed
  // q|k|v (3h) and FFN hidden (4h) share one region (q|k|v is consumed before
  // the self-attention barrier, the hidden written after the cross-attention
  // one); the pushed FFN output shares the normalised input's region (its last
  // local reader, the FFN's first mat-vec, is behind a barrier before any push)
  const size_t hm = multi ? (size_t)h : 0;
  L.mx = o;       o += al16(hm * 4);
  L.ma = o;       o += al16(hm * 4);
  L.mc = L.ma;
  L.mn = o;       o += al16(hm * 4);
  L.xo = L.mn;
  L.v3 = o;
  L.hb = o;       o += al16(4 * hm * 4);
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

// Sums of U independent per-lane values across the warp, reductions interleaved.
template <int U>
SP_DEVINL void warp_sum_n(float (&v)[U]) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
    for (int u = 0; u < U; ++u) v[u] += __shfl_xor_sync(0xffffffffu, v[u], o);
  }
}

// Block-wide sums of U values per thread (red: NW * U floats); every thread
// gets the totals, summed in warp order.
template <int U>
SP_DEVINL void block_sum_n(float (&v)[U], float* red) {
  warp_sum_n<U>(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  if (l == 0) {
#pragma unroll
    for (int u = 0; u < U; ++u) red[w * U + u] = v[u];
  }
  __syncthreads();
#pragma unroll
  for (int u = 0; u < U; ++u) {
    float t = 0.f;
#pragma unroll
    for (int k = 0; k < NW; ++k) t += red[k * U + u];
    v[u] = t;
  }
}

SP_DEVINL float dot4(const float4& a, const float4& b) { return a.x * b.x + a.y * b.y + a.z * b.z + a.w * b.w; }

// Keeps the best `keep` (value, index) pairs seen so far, best first, in a list
// of capacity GL.  All lanes of a warp hold the same list.
template <int GL>
SP_DEVINL void top_insert(float (&tv)[GL], int (&ti)[GL], float v, int j, int keep) {
  // the current last kept entry, selected with compile-time indices only so the
  // list stays in registers
  float lv = tv[0];
  int li = ti[0];
#pragma unroll
  for (int k = 1; k < GL; ++k) {
    if (k == keep - 1) {
      lv = tv[k];
      li = ti[k];
    }
  }
  if (!better(v, j, lv, li)) return;
#pragma unroll
  for (int k = GL - 1; k > 0; --k) {
    if (k < keep) {
      if (better(v, j, tv[k - 1], ti[k - 1])) {
        tv[k] = tv[k - 1];
        ti[k] = ti[k - 1];
      } else if (better(v, j, tv[k], ti[k])) {
        tv[k] = v;
        ti[k] = j;
      }
    }
  }
  if (better(v, j, tv[0], ti[0])) {
    tv[0] = v;
    ti[0] = j;
  }
}

// Order-preserving 32-bit key of a float (larger float -> larger key; -0 is
// taken as +0); 0 is reserved for "no entry".
SP_DEVINL uint32_t fkey(float v) {
  const uint32_t u = __float_as_uint(v + 0.0f);
  return (u >> 31) ? ~u : (u | 0x80000000u);
}
SP_DEVINL float fkey_inv(uint32_t k) {
  if (k == 0u) return -INFINITY;
  return __uint_as_float((k >> 31) ? (k & 0x7FFFFFFFu) : ~k);
}

// Warp-wide selection of the best `per` of `tot` contiguous (value, index)
// entries (value desc, index asc), E entries per lane at most; every lane gets
// the result, best first.  Each pick is two redux.sync reductions: the largest
// key, then the smallest index holding it.
template <int GL, int E>
SP_DEVINL void warp_merge_lists(const float* vin, const int* iin, int tot, int per, float (&out_v)[GL],
                                int (&out_i)[GL]) {
  const int lane = threadIdx.x & 31;
  uint32_t key[E];
  int ei[E];
#pragma unroll
  for (int k = 0; k < E; ++k) {
    const int idx = lane + 32 * k;
    key[k] = 0u;
    ei[k] = INT_MAX;
    if (idx < tot) {
      ei[k] = iin[idx];
      if (ei[k] != INT_MAX) key[k] = fkey(vin[idx]);
    }
  }
#pragma unroll
  for (int r = 0; r < GL; ++r) {
    out_v[r] = -INFINITY;
    out_i[r] = INT_MAX;
    if (r < per) {
      uint32_t bk = key[0];
      int bi = ei[0];
#pragma unroll
      for (int k = 1; k < E; ++k)
        if (key[k] > bk || (key[k] == bk && ei[k] < bi)) { bk = key[k]; bi = ei[k]; }
      const uint32_t mk = __reduce_max_sync(0xffffffffu, bk);
      const int mi = (int)__reduce_min_sync(0xffffffffu, bk == mk ? (uint32_t)bi : 0x7fffffffu);
      out_v[r] = fkey_inv(mk);
      out_i[r] = mk ? mi : INT_MAX;
#pragma unroll
      for (int k = 0; k < E; ++k)
        if (ei[k] == mi) { key[k] = 0u; ei[k] = INT_MAX; }
    }
  }
}

// HV = h / 128: float4 slices per lane of an h-vector (lane holds elements
// 4 (lane + 32 k) .. +3, k < HV).  GL = capacity of the per-round top lists
// (g + 1 <= GL).  P = history positions a warp loads at once.
// TRAIN: also accumulate the training pathway's aggregates along the rollout
// (Eqs. 5-7; g = 1 and keys in shared memory only): every CTA merges the C
// softmax partials (max, sum) of the round's available logits with STOP's in
// rank order, adds A_t beta^t p_t(j) to the scores of its own candidates and
// advances A_t and the soft count identically.
template <int HV, int GL, bool TRAIN, bool MULTI>
__global__ void __launch_bounds__(NT, 1)
select_kernel(const BatchDesc bd, const SelectArgs a, int n_loc_max, int keys_in_smem, int tm_cols) {
  constexpr int P = (16 / HV) > 0 ? 16 / HV : 1;
  constexpr int DPT = (HV * 128) / NT > 0 ? (HV * 128) / NT : 1;  // dims per thread in the merges
  constexpr int U = 4;                                          // candidates per warp iteration
  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int rank = (int)cluster.block_rank();
  const int e = blockIdx.x / C;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int h = a.h, k_max = a.k_max, g = a.g;
  const int per = g + 1;

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
  const SelSmem L = sel_layout(h, n_loc_max, k_max, C, keys_in_smem != 0, MULTI);
  float* kt_s = reinterpret_cast<float*>(sm + L.kt);
  float* lgp = reinterpret_cast<float*>(sm + L.lgp);
  float* stopkt = reinterpret_cast<float*>(sm + L.stopkt);
  float* wpart_o = reinterpret_cast<float*>(sm + L.wpart_o);
  float* wpart_ml = reinterpret_cast<float*>(sm + L.wpart_ml);
  float* all_o = reinterpret_cast<float*>(sm + L.all_o);
  float* all_ml = reinterpret_cast<float*>(sm + L.all_ml);
  float* wtop_v = reinterpret_cast<float*>(sm + L.wtop_v);
  int* wtop_i = reinterpret_cast<int*>(sm + L.wtop_i);
  float* all_tv = reinterpret_cast<float*>(sm + L.all_tv);
  int* all_ti = reinterpret_cast<int*>(sm + L.all_ti);
  float* xp_s = reinterpret_cast<float*>(sm + L.xp);
  uint8_t* taken = sm + L.taken;
  int* hist = reinterpret_cast<int*>(sm + L.hist);
  float* misc = reinterpret_cast<float*>(sm + L.misc);
  float* red = misc;                                  // [0, 16)  NW x 2
  float* gtop_v = misc + 64;                          // [64, 81)
  int* gtop_i = reinterpret_cast<int*>(misc + 96);    // [96, 113)
  uint32_t* tm_slot = reinterpret_cast<uint32_t*>(misc + 124);
  float* smx = misc + 20;                             // [20, 23) merged softmax: max, 1 / sum, p(STOP)
  float* wsm = reinterpret_cast<float*>(sm + L.wsm);
  float* all_sm = reinterpret_cast<float*>(sm + L.all_sm);
  float* score_s = reinterpret_cast<float*>(sm + L.score);

  // TMEM cache of the history rows this CTA attends over (tm_cols columns; 0 =
  // off): a key / value row is read from L2 once, in the round its position
  // joins the history, and from TMEM in every later round.  Warp w owns lanes
  // 32 (w % 4) .. +31 of columns [(w / 4) tm_cols / 2, +tm_cols / 2): ppw
  // positions of 8 HV columns each (key row, then value row, in the float4 lane
  // layout of the loads below).  The host sizes tm_cols so that every CTA that
  // can be resident on an SM gets its share of the 512 columns.
  if (tm_cols > 0 && warp == 0) {
    tmem_alloc(tm_slot, (uint32_t)tm_cols);
    tmem_relinquish();
  }

  // stage this CTA's slice of the folded keys and the STOP key
  const float* KT = a.KT;
  const int h4 = h >> 2;
  const int LD = n_loc_max + 1;  // columns of the dims-major key block
  if (keys_in_smem) {
    for (int i = tid; i < (nl + 1) * h4; i += NT) {
      const int j = i / h4, c = i % h4;
      const int row = (j < nl) ? row0 + j0 + j : a.stop_row;  // column nl: STOP
      reinterpret_cast<float4*>(kt_s)[(size_t)c * LD + j] =
          __ldg(reinterpret_cast<const float4*>(KT + (size_t)row * a.ldkt) + c);
    }
  }
  for (int i = tid; i < h4; i += NT)
    reinterpret_cast<float4*>(stopkt)[i] = __ldg(reinterpret_cast<const float4*>(KT + (size_t)a.stop_row * a.ldkt) + i);
  for (int j = tid; j < n_loc_max; j += NT) taken[j] = 0;
  if (TRAIN)
    for (int j = tid; j < n_loc_max; j += NT) score_s[j] = 0.f;
  if (tid == 0) hist[0] = a.start_row;
  const float bias = __ldg(a.stop_bias + e);
  const size_t trace = (size_t)e * (k_max + 1);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const int ppw = tm_cols / (16 * HV);  // cached positions per warp
  const uint32_t tm_base = tm_cols > 0 ? *tm_slot : 0u;
  const uint32_t tm_warp = tm_base + (((uint32_t)(warp & 3) * 32u) << 16) + (uint32_t)(warp >> 2) * (uint32_t)(tm_cols / 2);
  int np_cached = 0;  // history positions of this CTA already in TMEM

  // the per-element vectors of a round (residual, merged attention output,
  // LN2 output) are held DPT consecutive elements per thread
  auto el = [&](int d) { return tid * DPT + d; };
  // LN2 affine parameters, read once for the whole episode
  float g2[DPT], b2[DPT];
#pragma unroll
  for (int d = 0; d < DPT; ++d) {
    g2[d] = (a.ln2_g && el(d) < h) ? __ldg(a.ln2_g + el(d)) : 1.f;
    b2[d] = (a.ln2_b && el(d) < h) ? __ldg(a.ln2_b + el(d)) : 0.f;
  }
  // query / residual rows of the last history position, loaded one round ahead
  float zr[DPT];
  float4 q[HV];
  float shift;
  auto load_last = [&](int row) {
    const float* zrow = a.Z + (size_t)row * a.ldz;
    shift = __ldg(zrow);  // common shift of the LN moments (any value near the data)
#pragma unroll
    for (int d = 0; d < DPT; ++d) zr[d] = (el(d) < h) ? __ldg(zrow + el(d)) : 0.f;
    const float4* qrow = reinterpret_cast<const float4*>(a.QS + (size_t)row * a.ldqs);
#pragma unroll
    for (int k = 0; k < HV; ++k) q[k] = __ldg(qrow + lane + 32 * k);
  };
  if (!MULTI) load_last(a.start_row);

  // ---- decoders of several layers (MULTI): the layers before the last run on
  //      the new history position at the start of every round.  Every vector
  //      below is identical in all CTAs of the cluster (each product row is
  //      computed by one CTA and pushed to all; merges go in rank order).
  float* mx = reinterpret_cast<float*>(sm + L.mx);  // residual of the new position
  float* ma = reinterpret_cast<float*>(sm + L.ma);  // after self-attention
  float* mc = reinterpret_cast<float*>(sm + L.mc);  // after cross-attention
  float* mn = reinterpret_cast<float*>(sm + L.mn);  // a normalised input
  float* v3 = reinterpret_cast<float*>(sm + L.v3);  // pushed q | k | Wo Wv x
  float* hb = reinterpret_cast<float*>(sm + L.hb);  // pushed FFN hidden
  float* xo = reinterpret_cast<float*>(sm + L.xo);  // pushed FFN output
  const int ldc = 2 * h;
  float* ecache = MULTI ? a.dcache + (size_t)e * a.dcache_ep : nullptr;
  auto lcache = [&](int l) { return ecache + (size_t)(l - 1) * (k_max + 1) * ldc; };  // layers >= 1

  // LayerNorm of a shared h-vector into dst (same arithmetic in every CTA)
  auto ln_vec = [&](const float* src, const float* g, const float* bb, float* dst) {
    float v[DPT];
    float mom[2] = {0.f, 0.f};
    const float sh = src[0];
#pragma unroll
    for (int d = 0; d < DPT; ++d) {
      const int i = el(d);
      v[d] = i < h ? src[i] : 0.f;
      if (i < h) {
        const float c = v[d] - sh;
        mom[0] += c;
        mom[1] += c * c;
      }
    }
    block_sum_n<2>(mom, red);
    const float m1 = mom[0] / (float)h;
    const float mean = sh + m1;
    const float rstd = rsqrtf(fmaxf(mom[1] / (float)h - m1 * m1, 0.f) + a.ln_eps);
#pragma unroll
    for (int d = 0; d < DPT; ++d) {
      const int i = el(d);
      if (i < h) dst[i] = (v[d] - mean) * rstd * (g ? __ldg(g + i) : 1.f) + (bb ? __ldg(bb + i) : 0.f);
    }
    __syncthreads();
  };
  // rows [rank R / C, +R / C) of W [R, h] (fp32) times the shared vector x;
  // half a warp per row, MR rows per half-warp at a time (their loads in
  // flight together; each row's sum in the same order whatever MR is); each
  // result is pushed into dst[row] of every CTA
  constexpr int MR = 4;
  auto matvec_f32_push = [&](const float* W, int R, const float* x, float* dst) {
    const int Rc = R / C, r0 = rank * Rc, hl = lane & 15, hw = lane >> 4;
    const int cu = h / 4;  // float4 chunks per row
    const float4* x4 = reinterpret_cast<const float4*>(x);
    for (int rb = (warp * 2 + hw) * MR; rb < Rc; rb += NW * 2 * MR) {
      const float4* wr[MR];
#pragma unroll
      for (int i = 0; i < MR; ++i) wr[i] = reinterpret_cast<const float4*>(W + (size_t)(r0 + min(rb + i, Rc - 1)) * h);
      float sv[MR];
#pragma unroll
      for (int i = 0; i < MR; ++i) sv[i] = 0.f;
#pragma unroll 4
      for (int u = hl; u < cu; u += 16) {
        const float4 xv = x4[u];
        float4 wv[MR];
#pragma unroll
        for (int i = 0; i < MR; ++i) wv[i] = __ldg(wr[i] + u);
#pragma unroll
        for (int i = 0; i < MR; ++i) sv[i] += dot4(xv, wv[i]);
      }
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) {
#pragma unroll
        for (int i = 0; i < MR; ++i) sv[i] += __shfl_xor_sync(0xffffffffu, sv[i], o);
      }
      if (hl < C) {
#pragma unroll
        for (int i = 0; i < MR; ++i)
          if (rb + i < Rc) *cluster.map_shared_rank(dst + r0 + rb + i, hl) = sv[i];
      }
    }
  };
  // the same for W [R, K] in bf16, optionally through the exact GELU
  auto matvec_bf16_push = [&](const __nv_bfloat16* W, int R, int K, const float* x, float* dst, bool act) {
    const int Rc = R / C, r0 = rank * Rc, hl = lane & 15, hw = lane >> 4;
    const int cu = K / 8;  // 8-element chunks per row
    const float4* x4 = reinterpret_cast<const float4*>(x);
    for (int rb = (warp * 2 + hw) * MR; rb < Rc; rb += NW * 2 * MR) {
      const uint4* wr[MR];
#pragma unroll
      for (int i = 0; i < MR; ++i) wr[i] = reinterpret_cast<const uint4*>(W + (size_t)(r0 + min(rb + i, Rc - 1)) * K);
      float sv[MR];
#pragma unroll
      for (int i = 0; i < MR; ++i) sv[i] = 0.f;
#pragma unroll 4
      for (int u = hl; u < cu; u += 16) {
        const float4 xa = x4[2 * u], xb = x4[2 * u + 1];
        const float xs[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
        uint4 pw[MR];
#pragma unroll
        for (int i = 0; i < MR; ++i) pw[i] = __ldg(wr[i] + u);
#pragma unroll
        for (int i = 0; i < MR; ++i) {
          const uint32_t q[4] = {pw[i].x, pw[i].y, pw[i].z, pw[i].w};
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float2 f = unpack_bf16x2(q[k]);
            sv[i] += f.x * xs[2 * k] + f.y * xs[2 * k + 1];
          }
        }
      }
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) {
#pragma unroll
        for (int i = 0; i < MR; ++i) sv[i] += __shfl_xor_sync(0xffffffffu, sv[i], o);
      }
      if (act) {
#pragma unroll
        for (int i = 0; i < MR; ++i) sv[i] = gelu_erf(sv[i]);
      }
      if (hl < C) {
#pragma unroll
        for (int i = 0; i < MR; ++i)
          if (rb + i < Rc) *cluster.map_shared_rank(dst + r0 + rb + i, hl) = sv[i];
      }
    }
  };

  // this CTA's attention partial (max, sum, weighted values) from its warps'
  // partials, pushed into slot `slot` of every CTA (as in step 1 below)
  auto push_partial = [&](float4 (&o_w)[HV], float m_w, float l_w, int slot) {
#pragma unroll
    for (int k = 0; k < HV; ++k) reinterpret_cast<float4*>(wpart_o + warp * h)[lane + 32 * k] = o_w[k];
    if (lane == 0) {
      wpart_ml[warp * 2 + 0] = m_w;
      wpart_ml[warp * 2 + 1] = l_w;
    }
    __syncthreads();
    const float mwl = lane < NW ? wpart_ml[lane * 2] : -INFINITY;
    const float lwl = lane < NW ? wpart_ml[lane * 2 + 1] : 0.f;
    const float m_c = fkey_inv(__reduce_max_sync(0xffffffffu, fkey(mwl)));
    const float cwl = (mwl == -INFINITY) ? 0.f : __expf(mwl - m_c);
    const float l_c = warp_sum(cwl * lwl);
    float cw[NW];
#pragma unroll
    for (int w = 0; w < NW; ++w) cw[w] = __shfl_sync(0xffffffffu, cwl, w);
    float* sl = all_o + ((size_t)slot * C + rank) * h;
#pragma unroll
    for (int d = 0; d < DPT; ++d) {
      const int i = el(d);
      if (i >= h) continue;
      float acc = 0.f;
#pragma unroll
      for (int w = 0; w < NW; ++w) acc += cw[w] * wpart_o[w * h + i];
      for (int r = 0; r < C; ++r) *cluster.map_shared_rank(sl + i, r) = acc;
    }
    if (tid < C) {
      float* ml = cluster.map_shared_rank(all_ml + ((size_t)slot * C + rank) * 2, tid);
      ml[0] = m_c;
      ml[1] = l_c;
    }
  };
  // o / l of the C partials in slot `slot`, merged in rank order (DPT per thread)
  auto merge_slot = [&](int slot, float (&out)[DPT]) {
    const float mrl = lane < C ? all_ml[(slot * C + lane) * 2] : -INFINITY;
    const float lrl = lane < C ? all_ml[(slot * C + lane) * 2 + 1] : 0.f;
    const float m = fkey_inv(__reduce_max_sync(0xffffffffu, fkey(mrl)));
    const float wrl = (mrl == -INFINITY) ? 0.f : __expf(mrl - m);
    const float inv = 1.f / warp_sum(wrl * lrl);
    float wr[16];
#pragma unroll
    for (int r = 0; r < 16; ++r) wr[r] = __shfl_sync(0xffffffffu, wrl, r);
#pragma unroll
    for (int d = 0; d < DPT; ++d) {
      const int i = el(d);
      out[d] = 0.f;
      if (i >= h) continue;
      float o = 0.f;
#pragma unroll
      for (int r = 0; r < 16; ++r)
        if (r < C) o += wr[r] * all_o[((size_t)slot * C + r) * h + i];
      out[d] = o * inv;
    }
  };
  constexpr int PL = P > 1 ? P / 2 : 1;  // rows per warp batch in the deep-decoder loops
  // online-softmax update of a warp's partial with PL scored rows (fewer rows per batch than step 1:
  // these loops share the registers with the step-1 state)
  auto absorb = [&](const float (&sc)[PL], const float4 (&vr)[PL][HV], int valid, float& m_w, float& l_w,
                    float4 (&o_w)[HV]) {
#pragma unroll
    for (int pp = 0; pp < PL; ++pp) {
      if (pp < valid) {
        const float sv = sc[pp];
        const float mn2 = fmaxf(m_w, sv);
        const float cw = (m_w == -INFINITY) ? 0.f : __expf(m_w - mn2);
        const float ps = __expf(sv - mn2);
        l_w = l_w * cw + ps;
#pragma unroll
        for (int k = 0; k < HV; ++k) {
          o_w[k].x = o_w[k].x * cw + ps * vr[pp][k].x;
          o_w[k].y = o_w[k].y * cw + ps * vr[pp][k].y;
          o_w[k].z = o_w[k].z * cw + ps * vr[pp][k].z;
          o_w[k].w = o_w[k].w * cw + ps * vr[pp][k].w;
        }
        m_w = mn2;
      }
    }
  };
  // layer l's causal self-attention of the new position (query qv) over this
  // CTA's history positions rank, rank + C, ... < t; layer 0 reads the
  // candidates' precomputed rows, deeper layers the episode's cache
  auto self_attn_partial = [&](int l, const float4 (&qv)[HV], int t_len, int slot) {
    const int np2 = (rank < t_len) ? (t_len - 1 - rank) / C + 1 : 0;
    float m_w = -INFINITY, l_w = 0.f;
    float4 o_w[HV];
#pragma unroll
    for (int k = 0; k < HV; ++k) o_w[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int k0 = warp * PL; k0 < np2; k0 += NW * PL) {
      float4 kr[PL][HV], vr[PL][HV];
#pragma unroll
      for (int pp = 0; pp < PL; ++pp) {
        if (k0 + pp < np2) {
          const int pos = rank + (k0 + pp) * C;
          if (l == 0) {
            const int row = hist[pos];
            const float4* ks = reinterpret_cast<const float4*>(a.KS + (size_t)row * a.ldks);
            const float4* vt = reinterpret_cast<const float4*>(a.VT + (size_t)row * a.ldvt);
#pragma unroll
            for (int k = 0; k < HV; ++k) {
              kr[pp][k] = __ldg(ks + lane + 32 * k);
              vr[pp][k] = __ldg(vt + lane + 32 * k);
            }
          } else {
            const float4* cr = reinterpret_cast<const float4*>(lcache(l) + (size_t)pos * ldc);
#pragma unroll
            for (int k = 0; k < HV; ++k) {
              kr[pp][k] = __ldcg(cr + lane + 32 * k);
              vr[pp][k] = __ldcg(cr + h / 4 + lane + 32 * k);
            }
          }
        }
      }
      float sc[PL];
#pragma unroll
      for (int pp = 0; pp < PL; ++pp) {
        sc[pp] = 0.f;
        if (k0 + pp < np2) {
#pragma unroll
          for (int k = 0; k < HV; ++k) sc[pp] += dot4(qv[k], kr[pp][k]);
        }
      }
      warp_sum_n<PL>(sc);
      absorb(sc, vr, np2 - k0, m_w, l_w, o_w);
    }
    push_partial(o_w, m_w, l_w, slot);
  };
  // layer l's cross-attention of the normalised input mn over every row of the
  // episode's memory (this CTA's candidate slice; rank 0 adds the STOP row),
  // with the folded keys (Wq_c^T Wk_c m / sqrt h) and values (Wo_c Wv_c m)
  auto cross_partial = [&](int l, int slot) {
    float4 xv[HV];
#pragma unroll
    for (int k = 0; k < HV; ++k) xv[k] = reinterpret_cast<const float4*>(mn)[lane + 32 * k];
    const float* KCl = a.KC + (size_t)2 * l * h;
    const int ncand = nl + (rank == 0 ? 1 : 0);
    float m_w = -INFINITY, l_w = 0.f;
    float4 o_w[HV];
#pragma unroll
    for (int k = 0; k < HV; ++k) o_w[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int k0 = warp * PL; k0 < ncand; k0 += NW * PL) {
      float4 kr[PL][HV], vr[PL][HV];
#pragma unroll
      for (int pp = 0; pp < PL; ++pp) {
        if (k0 + pp < ncand) {
          const int jj = k0 + pp;
          const int row = jj < nl ? row0 + j0 + jj : a.stop_row;
          const float4* kc = reinterpret_cast<const float4*>(KCl + (size_t)row * a.ldz);
#pragma unroll
          for (int k = 0; k < HV; ++k) {
            kr[pp][k] = __ldg(kc + lane + 32 * k);
            vr[pp][k] = __ldg(kc + h / 4 + lane + 32 * k);
          }
        }
      }
      float sc[PL];
#pragma unroll
      for (int pp = 0; pp < PL; ++pp) {
        sc[pp] = 0.f;
        if (k0 + pp < ncand) {
#pragma unroll
          for (int k = 0; k < HV; ++k) sc[pp] += dot4(xv[k], kr[pp][k]);
        }
      }
      warp_sum_n<PL>(sc);
      absorb(sc, vr, ncand - k0, m_w, l_w, o_w);
    }
    push_partial(o_w, m_w, l_w, slot);
  };

  float alive = 1.f, disc = a.beta, kbar_acc = 0.f;  // A_t, beta^t, Eq. 7 (TRAIN)
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

    if constexpr (MULTI) {
      // ---- 0. the new history position (candidate row hist[t - 1]) through
      //      the layers before the last, then the last layer's q | k | Wo Wv x
      //      for it (exchange slots: self-attention 0, cross-attention 1; the
      //      pushed products are read before the next barrier and rewritten only
      //      after several more)
      const int p = t - 1;
      const int rn = hist[p];
      const int owner = p % C;  // the CTA whose share of positions holds p
      for (int i = tid; i < h; i += NT) mx[i] = __ldg(a.Z + (size_t)rn * a.ldz + i);
      __syncthreads();
      for (int l = 0; l + 1 < a.n_dec; ++l) {
        const DecLayerDev dl = a.dec[l];
        float4 qv[HV];
        if (l == 0) {
          const float4* qr = reinterpret_cast<const float4*>(a.QS + (size_t)rn * a.ldqs);
#pragma unroll
          for (int k = 0; k < HV; ++k) qv[k] = __ldg(qr + lane + 32 * k);
        } else {
          ln_vec(mx, dl.ln1_g, dl.ln1_b, mn);
          matvec_f32_push(dl.Wf, 3 * h, mn, v3);
          cluster.sync();
#pragma unroll
          for (int k = 0; k < HV; ++k) qv[k] = reinterpret_cast<const float4*>(v3)[lane + 32 * k];
          if (rank == owner) {
            float* dst = lcache(l) + (size_t)p * ldc;
            for (int i = tid; i < 2 * h; i += NT) dst[i] = v3[h + i];
          }
          __syncthreads();
        }
        self_attn_partial(l, qv, t, 0);
        cluster.sync();
        {
          float o[DPT];
          merge_slot(0, o);
#pragma unroll
          for (int d = 0; d < DPT; ++d)
            if (el(d) < h) ma[el(d)] = mx[el(d)] + o[d];
        }
        __syncthreads();
        ln_vec(ma, dl.ln2_g, dl.ln2_b, mn);
        cross_partial(l, 1);
        cluster.sync();
        {
          float o[DPT];
          merge_slot(1, o);
#pragma unroll
          for (int d = 0; d < DPT; ++d)
            if (el(d) < h) mc[el(d)] = ma[el(d)] + o[d];
        }
        __syncthreads();
        ln_vec(mc, dl.ln3_g, dl.ln3_b, mn);
        matvec_bf16_push(dl.W1, 4 * h, h, mn, hb, true);
        cluster.sync();
        matvec_bf16_push(dl.W2, h, 4 * h, hb, xo, false);
        cluster.sync();
        for (int i = tid; i < h; i += NT) mx[i] = mc[i] + xo[i];
        __syncthreads();
      }
      const DecLayerDev dl = a.dec[a.n_dec - 1];
      ln_vec(mx, dl.ln1_g, dl.ln1_b, mn);
      matvec_f32_push(dl.Wf, 3 * h, mn, v3);
      cluster.sync();
#pragma unroll
      for (int k = 0; k < HV; ++k) q[k] = reinterpret_cast<const float4*>(v3)[lane + 32 * k];
      shift = mx[0];
#pragma unroll
      for (int d = 0; d < DPT; ++d) zr[d] = (el(d) < h) ? mx[el(d)] : 0.f;
      if (rank == owner) {
        float* dst = lcache(a.n_dec - 1) + (size_t)p * ldc;
        for (int i = tid; i < 2 * h; i += NT) dst[i] = v3[h + i];
      }
      __syncthreads();
    }

    // ---- 1. partial causal self-attention of the last position (its query and
    //      residual rows were loaded at the end of the previous round); every
    //      history row of the round is loaded at once.
    const int np = (rank < t) ? (t - 1 - rank) / C + 1 : 0;  // positions rank, rank + C, ...
    float m_w = -INFINITY, l_w = 0.f;
    float4 o_w[HV];
#pragma unroll
    for (int k = 0; k < HV; ++k) o_w[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int jj = 0, k0 = warp * P; k0 < np; ++jj, k0 += NW * P) {
      float4 kr[P][HV], vr[P][HV];
      bool fresh[P];  // read from L2 this round, to be kept in TMEM
#pragma unroll
      for (int pp = 0; pp < P; ++pp) {
        const int o = jj * P + pp;  // warp-uniform, like k0 and np
        fresh[pp] = false;
        if (k0 + pp < np) {
          if (o < ppw && k0 + pp < np_cached) {
            const uint32_t ta = tm_warp + (uint32_t)(o * 8 * HV);
            tmem_ld_f4<HV>(ta, kr[pp]);
            tmem_ld_f4<HV>(ta + 4 * HV, vr[pp]);
          } else if (MULTI) {  // the last layer's rows of the episode cache, by position
            const float4* cr =
                reinterpret_cast<const float4*>(lcache(a.n_dec - 1) + (size_t)(rank + (k0 + pp) * C) * ldc);
#pragma unroll
            for (int k = 0; k < HV; ++k) {
              kr[pp][k] = __ldcg(cr + lane + 32 * k);
              vr[pp][k] = __ldcg(cr + h / 4 + lane + 32 * k);
            }
            fresh[pp] = o < ppw;
          } else {
            const int row = hist[rank + (k0 + pp) * C];
            const float4* ks = reinterpret_cast<const float4*>(a.KS + (size_t)row * a.ldks);
            const float4* vt = reinterpret_cast<const float4*>(a.VT + (size_t)row * a.ldvt);
#pragma unroll
            for (int k = 0; k < HV; ++k) {
              kr[pp][k] = __ldg(ks + lane + 32 * k);
              vr[pp][k] = __ldg(vt + lane + 32 * k);
            }
            fresh[pp] = o < ppw;
          }
        }
      }
      if (ppw > 0) {
        tmem_ld_wait();
#pragma unroll
        for (int pp = 0; pp < P; ++pp) {
          if (k0 + pp < np && jj * P + pp < ppw && k0 + pp < np_cached) {
            reg_fence_f4<HV>(kr[pp]);
            reg_fence_f4<HV>(vr[pp]);
          }
        }
      }
      float sc[P];
#pragma unroll
      for (int pp = 0; pp < P; ++pp) {
        sc[pp] = 0.f;
        if (k0 + pp < np) {
#pragma unroll
          for (int k = 0; k < HV; ++k) sc[pp] += dot4(q[k], kr[pp][k]);
        }
      }
      warp_sum_n<P>(sc);
#pragma unroll
      for (int pp = 0; pp < P; ++pp) {
        if (k0 + pp < np) {
          const float s = sc[pp];
          const float mn = fmaxf(m_w, s);
          const float cw = (m_w == -INFINITY) ? 0.f : __expf(m_w - mn);
          const float ps = __expf(s - mn);
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
#pragma unroll
      for (int pp = 0; pp < P; ++pp) {
        if (fresh[pp]) {
          const uint32_t ta = tm_warp + (uint32_t)((jj * P + pp) * 8 * HV);
          tmem_st_f4<HV>(ta, kr[pp]);
          tmem_st_f4<HV>(ta + 4 * HV, vr[pp]);
        }
      }
    }
    if (ppw > 0) tmem_st_wait();  // this round's rows are in TMEM before the next round reads them
    np_cached = np;
#pragma unroll
    for (int k = 0; k < HV; ++k) reinterpret_cast<float4*>(wpart_o + warp * h)[lane + 32 * k] = o_w[k];
    if (lane == 0) {
      wpart_ml[warp * 2 + 0] = m_w;
      wpart_ml[warp * 2 + 1] = l_w;
    }
    __syncthreads();
    {  // this CTA's partial from its warps' partials (warp order), pushed into
       // slot [buf][rank] of every CTA of the cluster
      // lane w holds warp w's (max, sum); one redux for the max, one warp sum
      const float mwl = lane < NW ? wpart_ml[lane * 2] : -INFINITY;
      const float lwl = lane < NW ? wpart_ml[lane * 2 + 1] : 0.f;
      const float m_c = fkey_inv(__reduce_max_sync(0xffffffffu, fkey(mwl)));
      const float cwl = (mwl == -INFINITY) ? 0.f : __expf(mwl - m_c);
      const float l_c = warp_sum(cwl * lwl);
      float cw[NW];
#pragma unroll
      for (int w = 0; w < NW; ++w) cw[w] = __shfl_sync(0xffffffffu, cwl, w);
      float* slot = all_o + ((size_t)buf * C + rank) * h;
      if (el(0) < h) {
        float acc[DPT];
#pragma unroll
        for (int d = 0; d < DPT; ++d) {
          acc[d] = 0.f;
#pragma unroll
          for (int w = 0; w < NW; ++w) acc[d] += cw[w] * wpart_o[w * h + el(d)];
        }
        // one vector store per peer (DPT consecutive elements)
        for (int r = 0; r < C; ++r) {
          float* dst = cluster.map_shared_rank(slot, r) + el(0);
          if (DPT == 4)
            *reinterpret_cast<float4*>(dst) = make_float4(acc[0], acc[DPT > 1 ? 1 : 0], acc[DPT > 2 ? 2 : 0],
                                                          acc[DPT > 3 ? 3 : 0]);
          else if (DPT == 2)
            *reinterpret_cast<float2*>(dst) = make_float2(acc[0], acc[DPT > 1 ? 1 : 0]);
          else
            dst[0] = acc[0];
        }
      }
      if (tid < C) {
        float* ml = cluster.map_shared_rank(all_ml + ((size_t)buf * C + rank) * 2, tid);
        ml[0] = m_c;
        ml[1] = l_c;
      }
    }
    cluster.sync();

    // ---- 2. merge the C partials (rank order, local reads), residual, LN2
    //      (one reduction of the moments shifted by z_last[0])
    // lane r holds CTA r's (max, sum); one redux for the max, one warp sum
    const float mrl = lane < C ? all_ml[(buf * C + lane) * 2] : -INFINITY;
    const float lrl = lane < C ? all_ml[(buf * C + lane) * 2 + 1] : 0.f;
    const float m = fkey_inv(__reduce_max_sync(0xffffffffu, fkey(mrl)));
    const float wrl = (mrl == -INFINITY) ? 0.f : __expf(mrl - m);
    const float wsum = warp_sum(wrl * lrl);
    float wr[16];
#pragma unroll
    for (int r = 0; r < 16; ++r) wr[r] = __shfl_sync(0xffffffffu, wrl, r);
    const float inv = 1.f / wsum;
    float uv[DPT];
    float mom[2] = {0.f, 0.f};
#pragma unroll
    for (int d = 0; d < DPT; ++d) {
      const int i = el(d);
      uv[d] = 0.f;
      if (i >= h) continue;
      float o = 0.f;
#pragma unroll
      for (int r = 0; r < 16; ++r)
        if (r < C) o += wr[r] * all_o[((size_t)buf * C + r) * h + i];
      uv[d] = zr[d] + o * inv;
      const float c = uv[d] - shift;
      mom[0] += c;
      mom[1] += c * c;
    }
    block_sum_n<2>(mom, red);
    const float m1 = mom[0] / (float)h;
    const float mean = shift + m1;
    const float rstd = rsqrtf(fmaxf(mom[1] / (float)h - m1 * m1, 0.f) + a.ln_eps);
#pragma unroll
    for (int d = 0; d < DPT; ++d) {
      const int i = el(d);
      if (i >= h) continue;
      xp_s[i] = (uv[d] - mean) * rstd * g2[d] + b2[d];
    }
    __syncthreads();

    // ---- 3. logits of the available local candidates (U per warp iteration,
    //      reductions interleaved), per-warp top g+1, and the raw STOP logit
    float4 xr[HV];
#pragma unroll
    for (int k = 0; k < HV; ++k) xr[k] = reinterpret_cast<const float4*>(xp_s)[lane + 32 * k];
    float tv[GL];
    int ti[GL];
#pragma unroll
    for (int k = 0; k < GL; ++k) { tv[k] = -INFINITY; ti[k] = INT_MAX; }
    float stop_raw;
    float vkeep = -INFINITY;  // this thread's candidate logit (keys in shared memory), -inf if unavailable
    if (keys_in_smem) {
      // dims-major keys: warp w takes a slice of the dims, lane = column
      // (candidates and, at column nl, STOP); per-warp partials are summed per
      // column in warp order, so every CTA computes STOP identically
      constexpr int JL = 4;  // columns per lane (nl + 1 <= 128)
      const float4* kt4 = reinterpret_cast<const float4*>(kt_s);
      const float4* xp4 = reinterpret_cast<const float4*>(xp_s);
      const int ncol = nl + 1;
      const int dper = h4 / NW;
      const int d0 = warp * dper;
      float acc[JL];
#pragma unroll
      for (int c = 0; c < JL; ++c) acc[c] = 0.f;
      for (int dd = 0; dd < dper; ++dd) {
        const float4 xv = xp4[d0 + dd];
        const float4* col = kt4 + (size_t)(d0 + dd) * LD;
#pragma unroll
        for (int c = 0; c < JL; ++c) {
          const int j = lane + 32 * c;
          if (j < ncol) acc[c] += dot4(xv, col[j]);
        }
      }
#pragma unroll
      for (int c = 0; c < JL; ++c) {
        const int j = lane + 32 * c;
        if (j < ncol) lgp[warp * LD + j] = acc[c];
      }
      __syncthreads();
      float sr = 0.f;
#pragma unroll
      for (int w = 0; w < NW; ++w) sr += lgp[w * LD + nl];
      stop_raw = sr;
      float v = -INFINITY;
      int id = INT_MAX;
      if (tid < nl && !taken[tid]) {
        float sj = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) sj += lgp[w * LD + tid];
        v = sj;
        id = j0 + tid;
      }
      vkeep = v;
      // this warp's top g+1 (one candidate per lane)
      uint32_t key = (id == INT_MAX) ? 0u : fkey(v);
#pragma unroll
      for (int r = 0; r < GL; ++r) {
        tv[r] = -INFINITY;
        ti[r] = INT_MAX;
        if (r < per) {
          const uint32_t mk = __reduce_max_sync(0xffffffffu, key);
          const int mi = (int)__reduce_min_sync(0xffffffffu, key == mk ? (uint32_t)id : 0x7fffffffu);
          tv[r] = fkey_inv(mk);
          ti[r] = mk ? mi : INT_MAX;
          if (id == mi) { key = 0u; id = INT_MAX; }
        }
      }
      if (TRAIN) {  // the warp's softmax partial relative to its best logit tv[0]
        const float ex = (vkeep != -INFINITY) ? expf((vkeep - tv[0]) * a.inv_tau) : 0.f;
        const float l_w = warp_sum(ex);
        if (lane == 0) {
          wsm[warp * 2] = tv[0];
          wsm[warp * 2 + 1] = l_w;
        }
      }
    } else {
      for (int jb = warp * U; jb < nl; jb += NW * U) {
        float sv[U];
        bool ok[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int j = jb + u;
          ok[u] = j < nl && !taken[j];
          sv[u] = 0.f;
          const float4* kr = reinterpret_cast<const float4*>(KT + (size_t)(row0 + j0 + min(j, nl - 1)) * a.ldkt);
#pragma unroll
          for (int k = 0; k < HV; ++k) sv[u] += dot4(xr[k], __ldg(kr + lane + 32 * k));
        }
        warp_sum_n<U>(sv);
#pragma unroll
        for (int u = 0; u < U; ++u)
          if (ok[u]) top_insert<GL>(tv, ti, sv[u], j0 + jb + u, per);
      }
      float s1[1] = {0.f};
#pragma unroll
      for (int k = 0; k < HV; ++k) s1[0] += dot4(xr[k], reinterpret_cast<const float4*>(stopkt)[lane + 32 * k]);
      warp_sum_n<1>(s1);
      stop_raw = s1[0];  // every warp of every CTA computes the same value
    }
    if (lane == 0) {
#pragma unroll
      for (int k = 0; k < GL; ++k) {
        if (k < per) {
          wtop_v[warp * per + k] = tv[k];
          wtop_i[warp * per + k] = ti[k];
        }
      }
    }
    __syncthreads();
    if (warp == 0) {  // CTA list from the warp lists, pushed into slot [buf][rank] of every CTA
      float cv[GL];
      int ci[GL];
      if (NW * per <= 32)
        warp_merge_lists<GL, 1>(wtop_v, wtop_i, NW * per, per, cv, ci);
      else
        warp_merge_lists<GL, 9>(wtop_v, wtop_i, NW * per, per, cv, ci);
      if (TRAIN) {  // the CTA's softmax partial, pushed with its list
        const float mw = lane < NW ? wsm[lane * 2] : -INFINITY;
        const float lw = lane < NW ? wsm[lane * 2 + 1] : 0.f;
        const float mc = fkey_inv(__reduce_max_sync(0xffffffffu, fkey(mw)));
        const float lc = warp_sum(mw == -INFINITY ? 0.f : lw * expf((mw - mc) * a.inv_tau));
        if (lane < C) {
          float* d = cluster.map_shared_rank(all_sm + ((size_t)buf * C + rank) * 2, lane);
          d[0] = mc;
          d[1] = lc;
        }
      }
      if (lane < C) {
        float* dv = cluster.map_shared_rank(all_tv + (size_t)buf * C * (GMAX + 1) + rank * per, lane);
        int* di = cluster.map_shared_rank(all_ti + (size_t)buf * C * (GMAX + 1) + rank * per, lane);
#pragma unroll
        for (int k = 0; k < GL; ++k) {
          if (k < per) {
            dv[k] = cv[k];
            di[k] = ci[k];
          }
        }
      }
    }
    cluster.sync();

    // ---- 4. merge the C lists (local reads, identically in every CTA) and decide
    if (warp == 0) {
      float gv[GL];
      int gi[GL];
      const float* lv = all_tv + (size_t)buf * C * (GMAX + 1);
      const int* li = all_ti + (size_t)buf * C * (GMAX + 1);
      if (C * per <= 32)
        warp_merge_lists<GL, 1>(lv, li, C * per, per, gv, gi);
      else
        warp_merge_lists<GL, 9>(lv, li, C * per, per, gv, gi);
      if (lane == 0) {
#pragma unroll
        for (int k = 0; k < GL; ++k) {
          if (k < per) {
            gtop_v[k] = gv[k];
            gtop_i[k] = gi[k];
          }
        }
      }
      if (TRAIN) {  // p_t = softmax(l_t / tau) over the available candidates and STOP
        const float sl = stop_raw + bias;
        const float mr = lane < C ? all_sm[((size_t)buf * C + lane) * 2] : -INFINITY;
        const float lr = lane < C ? all_sm[((size_t)buf * C + lane) * 2 + 1] : 0.f;
        const float mx = fmaxf(fkey_inv(__reduce_max_sync(0xffffffffu, fkey(mr))), sl);
        const float zv = warp_sum(mr == -INFINITY ? 0.f : lr * expf((mr - mx) * a.inv_tau));
        const float es = expf((sl - mx) * a.inv_tau);
        if (lane == 0) {
          smx[0] = mx;
          smx[1] = 1.f / (zv + es);
          smx[2] = es / (zv + es);
        }
      }
    }
    __syncthreads();
    if (TRAIN) {  // Eqs. 5-7 at this step (identical A_t in every CTA)
      const float ps = smx[2];
      if (vkeep != -INFINITY) score_s[tid] += alive * disc * (expf((vkeep - smx[0]) * a.inv_tau) * smx[1]);
      kbar_acc += alive * (1.f - ps);
      alive *= 1.f - ps;
      disc *= a.beta;
    }
    const float stop_logit = stop_raw + bias;
    const float best = gtop_v[0];
    if (rank == 0 && tid == 0) {
      if (a.gap) a.gap[trace + round] = best - stop_raw;
      if (a.margin) {
        // smallest gap between consecutive values among the top g+1 of
        // {available visual logits} U {STOP}
        float vals[GMAX + 2];
        int n = 0;
        const int nv = min(per, n_avail);
        for (int k = 0; k < nv; ++k) vals[n++] = gtop_v[k];
        int ins = n;
        while (ins > 0 && vals[ins - 1] < stop_logit) --ins;
        for (int k = n; k > ins; --k) vals[k] = vals[k - 1];
        vals[ins] = stop_logit;
        ++n;
        const int use = min(n, per);
        float mg = INFINITY;
        for (int k = 0; k + 1 < use; ++k) mg = fminf(mg, vals[k] - vals[k + 1]);
        a.margin[trace + round] = mg;
      }
    }
    ++round;
    if (stop_logit > best) break;  // STOP
    const int take = min(min(g, k_max - nsel), n_avail);
    if (tid < take) {
      const int jj = gtop_i[tid];
      if (jj < 0 || jj >= n_e) {
        set_error(a.err, SP_DEVERR_INDEX);
        hist[t + tid] = a.start_row;
      } else {
        hist[t + tid] = row0 + jj;
        if (jj >= j0 && jj < j0 + nl) taken[jj - j0] = 1;
        if (rank == 0 && a.order) a.order[(size_t)e * k_max + nsel + tid] = jj;
      }
    }
    {  // rows of the next round's last position
      const int jl = gtop_i[take - 1];
      if (!MULTI) load_last((jl >= 0 && jl < n_e) ? row0 + jl : a.start_row);
    }
    nsel += take;
    __syncthreads();
  }
  if (rank == 0 && tid == 0) {
    if (a.ep_count) a.ep_count[e] = nsel;
    if (a.rounds) a.rounds[e] = round;
    if (TRAIN) a.kbar[e] = kbar_acc;
  }
  if (TRAIN) {
    __syncthreads();
    for (int j = tid; j < nl; j += NT) a.score[row0 + j0 + j] = score_s[j];
  }
  tc_fence_before();
  cluster.sync();  // no CTA leaves while a peer may still write into it
  if (tm_cols > 0 && warp == 0) {
    tc_fence_after();
    tmem_dealloc(tm_base, (uint32_t)tm_cols);
  }
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

int select_cluster_size(const BatchDesc& bd, int h, int k_max, bool* keys_in_smem, size_t* smem_bytes, bool multi) {
  int n_max = 0;
  for (int b = 0; b < bd.B; ++b) {
    const int n = bd.vis_off[b + 1] - bd.vis_off[b];
    n_max = std::max(n_max, bd.group_size > 0 ? std::min(bd.group_size, n) : n);
  }
  const size_t budget = 225 * 1024;
  for (int C : {8, 16}) {
    const int n_loc = (n_max + C - 1) / C;
    const size_t need = sel_layout(h, n_loc, k_max, C, true, multi).total;
    if (n_loc + 1 <= 128 && need <= budget) {  // the dims-major logits take <= 128 columns
      *keys_in_smem = true;
      *smem_bytes = need;
      return C;
    }
  }
  *keys_in_smem = false;
  *smem_bytes = sel_layout(h, (n_max + 15) / 16, k_max, 16, false, multi).total;
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
  const SelSmem L = sel_layout(a.h, n_loc, a.k_max, C, keys_in_smem, a.n_dec > 1);
  void (*kern)(const BatchDesc, const SelectArgs, int, int, int) = nullptr;
  const int gl = a.g + 1 <= 2 ? 2 : (a.g + 1 <= 6 ? 6 : 17);
  const bool train = a.score != nullptr;
  if (train && (a.g != 1 || !keys_in_smem || !a.kbar)) return cudaErrorInvalidValue;
  const bool multi = a.n_dec > 1;
  if (multi && (a.g != 1 || train || !a.dec || !a.dcache || !a.KC)) return cudaErrorInvalidValue;
#define SP_SEL_CASE(HV_)                                                                                    \
  case HV_:                                                                                                 \
    kern = multi ? select_kernel<HV_, 2, false, true>                                                       \
                 : train ? select_kernel<HV_, 2, true, false>                                               \
                         : (gl == 2 ? select_kernel<HV_, 2, false, false>                                   \
                                    : (gl == 6 ? select_kernel<HV_, 6, false, false>                        \
                                               : select_kernel<HV_, 17, false, false>));                    \
    break;
  switch (a.h / 128) {
    SP_SEL_CASE(1)
    SP_SEL_CASE(2)
    SP_SEL_CASE(4)
    SP_SEL_CASE(8)
    default: return cudaErrorInvalidValue;
  }
#undef SP_SEL_CASE
  cudaError_t r = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L.total);
  if (r != cudaSuccess) return r;
  if (C > 8) {
    r = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (r != cudaSuccess) return r;
  }
  // TMEM history cache: 512 columns shared by the CTAs of this kernel that fit on
  // one SM (so an allocation never waits on another cluster's CTA), at least
  // one position (16 HV columns for the two rows) per warp, else off
  int per_sm = 0;
  r = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, NT, L.total);
  if (r != cudaSuccess) return r;
  int tm_cols = 512;
  while (per_sm > 1 && tm_cols * per_sm > 512) tm_cols >>= 1;
  if (per_sm < 1 || tm_cols < 32 || tm_cols < 16 * (a.h / 128)) tm_cols = 0;
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
  r = cudaLaunchKernelEx(&cfg, kern, bd, a, n_loc, keys_in_smem ? 1 : 0, tm_cols);
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
