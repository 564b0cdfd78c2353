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

// Attention of the new token of every sequence over its cache (split keys,
// after flash-decoding): CTA (s, kvh, b) takes key range s of the L = lens[b]
// + 1 positions of sequence b (split into up to gridDim.x ranges of about
// DEC_CH keys) for the G = Hq / Hkv query heads sharing kv head kvh, so each
// cached row is read once.  Per DEC_CH-key tile: K and V rows to shared
// memory by bulk copies (one per row; position lens[b] is the new token's
// row, taken from qkv), scores G x DEC_CH (thread = key), online softmax in
// the exp2 domain, P V with a thread per pair of head dims and a quarter or
// half of the keys.  The range holding position lens[b] also appends the new
// key / value row to the cache.  With one range the CTA writes the output;
// else it writes (m, l, o) and the last range to finish (a counter per
// (b, kvh)) merges the ranges in range order.
constexpr int DEC_CH = 64;
constexpr int DEC_GMAX = 8;

template <int DH, int G>
__global__ void __launch_bounds__(128) decode_attn_split_kernel(
    const __nv_bfloat16* __restrict__ qkv, int ld_qkv, int kcol, int vcol, __nv_bfloat16* __restrict__ kv_l,
    int S_cap, const int* __restrict__ lens, int B, int Hkv, float* __restrict__ part, int* __restrict__ cnt,
    __nv_bfloat16* __restrict__ out, int ld_out, float scale_log2, int* err) {
  constexpr int RS = DH * 2 + 16;  // padded tile row (bytes): 16-byte reads of consecutive rows hit distinct banks
  constexpr int CPR = DH / 8;      // 16-byte chunks per row
  constexpr int DP = DH / 2;       // P V threads per key group (a pair of dims each)
  constexpr int KH = 128 / DP;     // key groups of the P V threads
  constexpr int KPG = DEC_CH / KH; // keys per group in a tile
  __shared__ __align__(16) uint8_t Ks[DEC_CH * RS];
  __shared__ __align__(16) uint8_t Vs[DEC_CH * RS];
  __shared__ __align__(16) float q_s[G * DH];
  __shared__ __align__(16) float p_s[G * DEC_CH];
  __shared__ __align__(16) float2 f_s[(KH - 1) * G * DP];
  __shared__ float m_s[G], l_s[G], c_s[G];
  __shared__ __align__(8) uint64_t bar;
  __shared__ int last_s;
  const int s = blockIdx.x, kvh = blockIdx.y, b = blockIdx.z;
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  if (t == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  pdl_wait();
  pdl_trigger();
  const int len = __ldg(lens + b);
  if (len < 0 || len >= S_cap) {
    if (t == 0 && s == 0 && kvh == 0) set_error(err, SP_DEVERR_INDEX);
    return;
  }
  const int L = len + 1;
  const int ns = min((int)gridDim.x, (L + DEC_CH - 1) / DEC_CH);
  if (s >= ns) return;
  const int k0 = (int)((long long)s * L / ns), k1 = (int)((long long)(s + 1) * L / ns);
  const int W = Hkv * DH;
  const __nv_bfloat16* qrow = qkv + (size_t)b * ld_qkv;
  const __nv_bfloat16* newk = qrow + kcol + kvh * DH;
  const __nv_bfloat16* newv = qrow + vcol + kvh * DH;
  __nv_bfloat16* Kc = kv_l + (size_t)b * S_cap * W + kvh * DH;
  __nv_bfloat16* Vc = kv_l + (size_t)(B + b) * S_cap * W + kvh * DH;
  if (len >= k0 && len < k1) {  // cache append (other ranges read positions < len only)
    for (int i = t; i < 2 * CPR; i += 128) {
      const bool isv = i >= CPR;
      const int c = isv ? i - CPR : i;
      reinterpret_cast<uint4*>((isv ? Vc : Kc) + (size_t)len * W)[c] =
          __ldg(reinterpret_cast<const uint4*>(isv ? newv : newk) + c);
    }
  }
  for (int i = t; i < G * DH; i += 128) q_s[i] = __bfloat162float(qrow[kvh * G * DH + i]);
  if (t < G) {
    m_s[t] = -INFINITY;
    l_s[t] = 0.f;
  }
  const int dp = t % DP, kh = t / DP;
  float2 o[G];
#pragma unroll
  for (int g = 0; g < G; ++g) o[g] = make_float2(0.f, 0.f);

  uint32_t phase = 0;
  for (int j0 = k0; j0 < k1; j0 += DEC_CH, phase ^= 1u) {
    const int nk = min(DEC_CH, k1 - j0);
    if (t == 0) mbar_arrive_expect_tx(&bar, (uint32_t)(2 * nk * DH * 2));
    __syncthreads();  // expect_tx before the copies; the previous tile's readers are done
    if (t < 2 * nk) {
      const bool isv = t >= nk;
      const int r = isv ? t - nk : t;
      const int p = j0 + r;
      const __nv_bfloat16* src = p < len ? (isv ? Vc : Kc) + (size_t)p * W : (isv ? newv : newk);
      bulk_g2s((isv ? Vs : Ks) + r * RS, src, DH * 2, &bar);
    }
    const bool ok = mbar_wait(&bar, phase, err);  // bounded; a timeout sets the error word
    if (__syncthreads_or(!ok)) return;
    for (int i = t; i < G * DEC_CH; i += 128) {
      const int g = i / DEC_CH, j = i - g * DEC_CH;
      float sc = -INFINITY;
      if (j < nk) {
        const uint4* kr = reinterpret_cast<const uint4*>(Ks + j * RS);
        const float4* qg = reinterpret_cast<const float4*>(q_s + g * DH);
        float acc = 0.f;
#pragma unroll
        for (int c = 0; c < CPR; ++c) {
          const uint4 u = kr[c];
          const float4 qa = qg[2 * c], qb = qg[2 * c + 1];
          float2 f = unpack_bf16x2(u.x);
          acc += f.x * qa.x + f.y * qa.y;
          f = unpack_bf16x2(u.y);
          acc += f.x * qa.z + f.y * qa.w;
          f = unpack_bf16x2(u.z);
          acc += f.x * qb.x + f.y * qb.y;
          f = unpack_bf16x2(u.w);
          acc += f.x * qb.z + f.y * qb.w;
        }
        sc = acc * scale_log2;
      }
      p_s[i] = sc;
    }
    __syncthreads();
    for (int g = warp; g < G; g += 4) {
      const float a = p_s[g * DEC_CH + lane], c = p_s[g * DEC_CH + lane + 32];
      const float mo = m_s[g];
      const float mn = fmaxf(mo, warp_max(fmaxf(a, c)));
      const float pa = exp2f(a - mn), pc = exp2f(c - mn);
      const float corr = (mo == -INFINITY) ? 0.f : exp2f(mo - mn);
      const float sum = warp_sum(pa + pc);
      p_s[g * DEC_CH + lane] = pa;
      p_s[g * DEC_CH + lane + 32] = pc;
      __syncwarp();
      if (lane == 0) {
        m_s[g] = mn;
        l_s[g] = l_s[g] * corr + sum;
        c_s[g] = corr;
      }
    }
    __syncthreads();
#pragma unroll
    for (int g = 0; g < G; ++g) {
      o[g].x *= c_s[g];
      o[g].y *= c_s[g];
    }
    const int ja = kh * KPG, jb = min(nk, ja + KPG);
#pragma unroll 4
    for (int j = ja; j < jb; ++j) {
      const float2 v = unpack_bf16x2(*reinterpret_cast<const uint32_t*>(Vs + j * RS + dp * 4));
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float pj = p_s[g * DEC_CH + j];
        o[g].x += pj * v.x;
        o[g].y += pj * v.y;
      }
    }
  }
  // fold the key groups into group 0 (fixed order)
  if (kh > 0) {
#pragma unroll
    for (int g = 0; g < G; ++g) f_s[((kh - 1) * G + g) * DP + dp] = o[g];
  }
  __syncthreads();
  if (kh == 0) {
#pragma unroll
    for (int q = 0; q < KH - 1; ++q)
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float2 x = f_s[(q * G + g) * DP + dp];
        o[g].x += x.x;
        o[g].y += x.y;
      }
  }
  const int h0 = kvh * G;
  const int Hq = Hkv * G;
  if (ns == 1) {
    if (kh == 0) {
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float il = 1.f / l_s[g];
        *reinterpret_cast<uint32_t*>(out + (size_t)b * ld_out + (h0 + g) * DH + 2 * dp) =
            pack_bf16x2(o[g].x * il, o[g].y * il);
      }
    }
    return;
  }
  // partial of this range: [b][h][range] x (o[DH], m, l)
  constexpr int STRIDE = DH + 2;
  if (kh == 0) {
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float* pp = part + (((size_t)b * Hq + h0 + g) * gridDim.x + s) * STRIDE;
      *reinterpret_cast<float2*>(pp + 2 * dp) = o[g];
      if (dp == 0) *reinterpret_cast<float2*>(pp + DH) = make_float2(m_s[g], l_s[g]);
    }
  }
  __syncthreads();
  if (t == 0) {
    __threadfence();
    last_s = atomicAdd(cnt + (size_t)b * Hkv + kvh, 1) == ns - 1;
  }
  __syncthreads();
  if (!last_s) return;
  __threadfence();
  if (kh == 0) {
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const float* pp = part + ((size_t)b * Hq + h0 + g) * gridDim.x * STRIDE;
      float mm = -INFINITY;
      for (int r = 0; r < ns; ++r) mm = fmaxf(mm, __ldcg(pp + r * STRIDE + DH));
      float nx = 0.f, ny = 0.f, den = 0.f;
      for (int r = 0; r < ns; ++r) {
        const float2 ml = __ldcg(reinterpret_cast<const float2*>(pp + r * STRIDE + DH));
        const float c = (ml.x == -INFINITY) ? 0.f : exp2f(ml.x - mm);
        const float2 x = __ldcg(reinterpret_cast<const float2*>(pp + r * STRIDE + 2 * dp));
        nx += c * x.x;
        ny += c * x.y;
        den += c * ml.y;
      }
      const float il = 1.f / den;
      *reinterpret_cast<uint32_t*>(out + (size_t)b * ld_out + (h0 + g) * DH + 2 * dp) = pack_bf16x2(nx * il, ny * il);
    }
  }
}

template <int DH, int G>
cudaError_t launch_decode_attn(dim3 grid, cudaStream_t st, const __nv_bfloat16* q, int ld, int kcol, int vcol,
                               __nv_bfloat16* kv, int S_cap, const int* lens, int B, int Hkv, float* part, int* cnt,
                               __nv_bfloat16* o, int ld_out, float sl2, int* err) {
  return launch_pdl(decode_attn_split_kernel<DH, G>, grid, dim3(128), 0, st, q, ld, kcol, vcol, kv, S_cap, lens, B,
                    Hkv, part, cnt, o, ld_out, sl2, err);
}

template <int DH>
cudaError_t dispatch_decode_attn(int G, dim3 grid, cudaStream_t st, const __nv_bfloat16* q, int ld, int kcol,
                                 int vcol, __nv_bfloat16* kv, int S_cap, const int* lens, int B, int Hkv,
                                 float* part, int* cnt, __nv_bfloat16* o, int ld_out, float sl2, int* err) {
#define SP_DEC_G(GG)                                                                                        \
  case GG:                                                                                                  \
    return launch_decode_attn<DH, GG>(grid, st, q, ld, kcol, vcol, kv, S_cap, lens, B, Hkv, part, cnt, o, \
                                      ld_out, sl2, err);
  switch (G) {
    SP_DEC_G(1) SP_DEC_G(2) SP_DEC_G(3) SP_DEC_G(4) SP_DEC_G(5) SP_DEC_G(6) SP_DEC_G(7) SP_DEC_G(8)
    default: return cudaErrorInvalidValue;
  }
#undef SP_DEC_G
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

size_t decode_attention_floats(int B, int Hq, int dh, int max_splits) {
  return (size_t)B * Hq * max_splits * (dh + 2);
}

cudaError_t decode_attention(const void* qkv, void* kv_l, int S_cap, const int* lens, int B, int Hq, int Hkv, int dh,
                             int max_len, float* part, int max_splits, int* cnt, void* out, int* err,
                             cudaStream_t st) {
  if (Hkv < 1 || Hq % Hkv != 0 || Hq / Hkv > DEC_GMAX || max_splits < 1) return cudaErrorInvalidValue;
  const int ld = (Hq + 2 * Hkv) * dh;
  const float sl2 = 1.4426950408889634f / sqrtf((float)dh);
  // ranges per sequence: one per DEC_CH keys of the longest sequence, at most max_splits
  const int ns = std::max(1, std::min(max_splits, (std::min(max_len, S_cap) + DEC_CH - 1) / DEC_CH));
  dim3 grid(ns, Hkv, B);
  const auto* q = reinterpret_cast<const __nv_bfloat16*>(qkv);
  auto* kv = reinterpret_cast<__nv_bfloat16*>(kv_l);
  auto* o = reinterpret_cast<__nv_bfloat16*>(out);
  prof_begin_launch(st);
  cudaError_t r;
  if (dh == 128)
    r = dispatch_decode_attn<128>(Hq / Hkv, grid, st, q, ld, Hq * dh, (Hq + Hkv) * dh, kv, S_cap, lens, B, Hkv,
                                  part, cnt, o, Hq * dh, sl2, err);
  else if (dh == 64)
    r = dispatch_decode_attn<64>(Hq / Hkv, grid, st, q, ld, Hq * dh, (Hq + Hkv) * dh, kv, S_cap, lens, B, Hkv,
                                 part, cnt, o, Hq * dh, sl2, err);
  else
    return cudaErrorInvalidValue;
  prof_end_launch(st, SP_K_ATTN, 0.0, 0.0);
  if (r != cudaSuccess) return r;
  return cudaGetLastError();
}

cudaError_t lens_increment(int* lens, int* rope_pos, int B, int S_cap, cudaStream_t st) {
  lens_increment_kernel<<<(B + 127) / 128, 128, 0, st>>>(lens, rope_pos, B, S_cap);
  return cudaGetLastError();
}

}  // namespace sp
