// The C ABI of libstepprune (include/stepprune.h): argument validation,
// workspace carving, tensor-map encoding and the sequencing of the kernels of
// every stage on the caller's stream.  No entry point allocates device memory
// except the *_create functions; no entry point synchronises the host except
// *_create and sp_profile_end.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "internal.h"

namespace sp {

// ------------------------------------------------------------------ errors

static thread_local std::string g_last_error;

static sp_status fail(sp_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

static sp_status cuda_fail(cudaError_t e, const char* where) {
  return fail(SP_ERR_CUDA, "%s: %s (%d)", where, cudaGetErrorString(e), (int)e);
}

#define SP_CUDA(call, where)                      \
  do {                                            \
    cudaError_t e__ = (call);                     \
    if (e__ != cudaSuccess) return cuda_fail(e__, where); \
  } while (0)

static bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// ------------------------------------------------------------------ device info

int device_sm_count() {
  static int cached_dev = -1, cached = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev != cached_dev) {
    cudaDeviceGetAttribute(&cached, cudaDevAttrMultiProcessorCount, dev);
    cached_dev = dev;
  }
  return cached > 0 ? cached : 1;
}

static sp_status check_device() {
  int dev = 0, major = 0, minor = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10 || minor != 3)
    return fail(SP_ERR_UNSUPPORTED, "device %d is sm_%d%d; this library is built for sm_103a only", dev,
                major, minor);
  return SP_OK;
}

// ------------------------------------------------------------------ tensor maps

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn(std::string* msg) {
  static EncodeTiledFn fn = nullptr;
  if (fn) return fn;
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q);
  if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !p) {
    if (msg) *msg = "cuTensorMapEncodeTiled is not available from the driver";
    return nullptr;
  }
  fn = reinterpret_cast<EncodeTiledFn>(p);
  return fn;
}

bool encode_tmap_bf16(CUtensorMap* map, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows,
                      std::string* msg) {
  EncodeTiledFn fn = encode_fn(msg);
  if (!fn) return false;
  if (rows == 0) rows = 1;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) {
      char b[160];
      snprintf(b, sizeof(b), "cuTensorMapEncodeTiled failed (%d) for %llux%llu box %u", (int)r,
               (unsigned long long)rows, (unsigned long long)cols, box_rows);
      *msg = b;
    }
    return false;
  }
  return true;
}

bool encode_tmap_2d(CUtensorMap* map, const void* ptr, bool f32, uint64_t rows, uint64_t cols,
                    uint32_t box_cols, uint32_t box_rows, std::string* msg) {
  EncodeTiledFn fn = encode_fn(msg);
  if (!fn) return false;
  if (rows == 0) rows = 1;
  const uint64_t es = f32 ? 4 : 2;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * es};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                  const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) {
      char b[160];
      snprintf(b, sizeof(b), "cuTensorMapEncodeTiled failed (%d) for %llux%llu box %ux%u", (int)r,
               (unsigned long long)rows, (unsigned long long)cols, box_cols, box_rows);
      *msg = b;
    }
    return false;
  }
  return true;
}

// ------------------------------------------------------------------ profiling

namespace {
struct Prof {
  bool on = false;
  int cap = 0, n = 0;
  std::vector<cudaEvent_t> ev;
  std::vector<int> kind;
  std::vector<double> flops, bytes;
};
Prof g_prof;
}  // namespace

bool prof_enabled() { return g_prof.on; }

void prof_begin_launch(cudaStream_t st) {
  if (!g_prof.on || g_prof.n >= g_prof.cap) return;
  cudaEventRecord(g_prof.ev[2 * g_prof.n], st);
}

void prof_end_launch(cudaStream_t st, int kind, double flops, double bytes) {
  if (!g_prof.on || g_prof.n >= g_prof.cap) return;
  cudaEventRecord(g_prof.ev[2 * g_prof.n + 1], st);
  g_prof.kind[g_prof.n] = kind;
  g_prof.flops[g_prof.n] = flops;
  g_prof.bytes[g_prof.n] = bytes;
  ++g_prof.n;
}

// ------------------------------------------------------------------ batches

bool pdl_enabled() {
  static const bool on = [] {
    const char* v = std::getenv("SP_PDL");
    return !(v && v[0] == '0');
  }();
  return on;
}

bool fill_batch_desc(BatchDesc* d, int B, const int* n_vis, const int* n_txt, int group_size,
                     std::string* msg) {
  if (B < 1 || B > SP_MAX_BATCH) {
    if (msg) *msg = "B must be in 1..SP_MAX_BATCH";
    return false;
  }
  if (!n_vis || !n_txt) {
    if (msg) *msg = "n_vis / n_txt are required host arrays";
    return false;
  }
  if (group_size < 0) {
    if (msg) *msg = "group_size must be >= 0";
    return false;
  }
  memset(d, 0, sizeof(*d));
  d->B = B;
  d->group_size = group_size;
  for (int b = 0; b < B; ++b) {
    if (n_vis[b] < 1 || n_vis[b] > SP_MAX_NVIS || n_txt[b] < 0) {
      if (msg) *msg = "n_vis[b] must be in 1..SP_MAX_NVIS and n_txt[b] >= 0";
      return false;
    }
    const int gs = group_size > 0 ? group_size : n_vis[b];
    d->vis_off[b + 1] = d->vis_off[b] + n_vis[b];
    d->txt_off[b + 1] = d->txt_off[b] + n_txt[b];
    d->ep_off[b + 1] = d->ep_off[b] + (n_vis[b] + gs - 1) / gs;
  }
  return true;
}

// Bump allocator over the caller's workspace (256-byte aligned slices).
struct Carve {
  char* base;
  size_t off = 0;
  explicit Carve(void* p) : base(static_cast<char*>(p)) {}
  template <class T>
  T* take(size_t n) {
    off = (off + 255) & ~size_t(255);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += n * sizeof(T);
    return p;
  }
};

}  // namespace sp

using namespace sp;

// ======================================================================= ABI

struct sp_selector_s {
  sp_selector_cfg cfg;
  sp_selector_weights w;
  // candidate precompute weights as six bf16 segments b0 b1 b0 b2 b1 b0 of
  //   Wcat1 [2h, D]: rows W_in | Wq_p^T Wk_p / sqrt(h)
  //   Wcat2 [3h, h]: rows Wq_s / sqrt(h) | Wk_s | Wo_s Wv_s
  void* P1s = nullptr;  // [2h, 6D]
  void* P2s = nullptr;  // [3h, 6h]
  GemmB P1, P2;
  GemmB Wp;
  // decoders of several layers: Wcat1 also holds, per layer before the last,
  // Wq_c^T Wk_c / sqrt(h) | Wo_c Wv_c; the runtime weights of layers >= 1
  int n_dec = 1;
  const float* pre_ln1_g = nullptr;  // layer 0's LN1 (applied in the precompute)
  const float* pre_ln1_b = nullptr;
  float* Wf = nullptr;               // [n_dec - 1][3h, h]
  DecLayerDev* dec_dev = nullptr;    // [n_dec]
  GemmB enc_qkv[SP_MAX_ENC_LAYERS], enc_o[SP_MAX_ENC_LAYERS], enc_1[SP_MAX_ENC_LAYERS],
      enc_2[SP_MAX_ENC_LAYERS];
};

struct sp_model_s {
  sp_model_cfg cfg;
  sp_model_weights w;
  float2* rope = nullptr;  // [max_pos, head_dim / 2]
  std::vector<GemmB> qkv, o, gu, down;
  GemmB p1, p2;
};

extern "C" {

const char* sp_last_error(void) { return g_last_error.c_str(); }
int sp_abi_version(void) { return SP_ABI_VERSION; }

sp_status sp_device_error_status(int w) {
  if (w == 0) return SP_OK;
  if (w & SP_DEVERR_TIMEOUT) return fail(SP_ERR_TIMEOUT, "a bounded device wait ran out (error word 0x%x)", w);
  return fail(SP_ERR_DEVICE, "device-side check failed (error word 0x%x)", w);
}

int sp_num_episodes(int B, const int* n_vis, int group_size) {
  if (B < 1 || B > SP_MAX_BATCH || !n_vis || group_size < 0) return -1;
  int e = 0;
  for (int b = 0; b < B; ++b) {
    if (n_vis[b] < 1) return -1;
    const int gs = group_size > 0 ? group_size : n_vis[b];
    e += (n_vis[b] + gs - 1) / gs;
  }
  return e;
}

int sp_packed_cap(int B, const int* n_vis, const int* n_txt, int k_cap) {
  if (B < 1 || B > SP_MAX_BATCH || !n_vis || !n_txt || k_cap < 0) return -1;
  long t = 0;
  for (int b = 0; b < B; ++b) {
    if (n_vis[b] < 1 || n_txt[b] < 0) return -1;
    t += std::min(n_vis[b], k_cap) + n_txt[b];
  }
  return t > 0x7fffffff ? -1 : (int)t;
}

// ------------------------------------------------------------------ selector

sp_status sp_selector_create(const sp_selector_cfg* cfg, const sp_selector_weights* w, sp_selector** out) {
  if (!cfg || !w || !out) return fail(SP_ERR_INVALID_ARG, "sp_selector_create: NULL argument");
  *out = nullptr;
  sp_status st = check_device();
  if (st != SP_OK) return st;
  const sp_selector_cfg c = *cfg;
  if (c.D <= 0 || c.D % 128 != 0) return fail(SP_ERR_SHAPE, "D must be a positive multiple of 128");
  if (c.h < 128 || c.h > 1024 || c.h % 128 != 0) return fail(SP_ERR_SHAPE, "h must be a multiple of 128 in 128..1024");
  if (c.n_enc_layers < 0 || c.n_enc_layers > SP_MAX_ENC_LAYERS) return fail(SP_ERR_SHAPE, "n_enc_layers out of range");
  if (c.n_enc_layers > 0) {
    if (c.D_text <= 0 || c.D_text % 64 != 0) return fail(SP_ERR_SHAPE, "D_text must be a multiple of 64");
    if (c.enc_head_dim != 64 && c.enc_head_dim != 128) return fail(SP_ERR_SHAPE, "enc_head_dim must be 64 or 128");
    if (c.D % c.enc_head_dim != 0) return fail(SP_ERR_SHAPE, "D must be a multiple of enc_head_dim");
    if (c.enc_ffn <= 0 || c.enc_ffn % 128 != 0) return fail(SP_ERR_SHAPE, "enc_ffn must be a multiple of 128");
    if (!w->W_p) return fail(SP_ERR_INVALID_ARG, "W_p is required with an encoder");
    for (int i = 0; i < c.n_enc_layers; ++i)
      if (!w->enc_wqkv[i] || !w->enc_wo[i] || !w->enc_w1[i] || !w->enc_w2[i])
        return fail(SP_ERR_INVALID_ARG, "encoder layer %d weights missing", i);
  }
  if (!(c.ln_eps > 0.f)) return fail(SP_ERR_INVALID_ARG, "ln_eps must be > 0");
  if (!w->s_stop || !w->s_start || !w->W_in || !w->Wq_s || !w->Wk_s || !w->Wv_s || !w->Wo_s || !w->Wq_p || !w->Wk_p)
    return fail(SP_ERR_INVALID_ARG, "pointer-decoder weights missing");
  const int nd = c.n_dec_layers <= 0 ? 1 : c.n_dec_layers;
  if (nd > SP_MAX_DEC_LAYERS) return fail(SP_ERR_SHAPE, "n_dec_layers must be in 1..SP_MAX_DEC_LAYERS");
  if (nd > 1 && !w->dec_lower) return fail(SP_ERR_INVALID_ARG, "dec_lower is required with n_dec_layers > 1");
  for (int l = 0; l + 1 < nd; ++l) {
    const sp_dec_layer_weights& L = w->dec_lower[l];
    if (!L.Wq_s || !L.Wk_s || !L.Wv_s || !L.Wo_s || !L.Wq_c || !L.Wo_c || !L.Wk_c || !L.Wv_c || !L.W1 || !L.W2)
      return fail(SP_ERR_INVALID_ARG, "decoder layer %d weights missing", l);
    if ((reinterpret_cast<uintptr_t>(L.W1) | reinterpret_cast<uintptr_t>(L.W2)) & 15)
      return fail(SP_ERR_ALIGN, "decoder layer %d: W1 / W2 must be 16-byte aligned", l);
  }

  sp_selector* s = new (std::nothrow) sp_selector_s();
  if (!s) return fail(SP_ERR_INVALID_ARG, "out of host memory");
  s->cfg = c;
  s->w = *w;
  const int h = c.h, D = c.D;
  const sp_dec_layer_weights* low = nd > 1 ? w->dec_lower : nullptr;
  s->n_dec = nd;
  // layer 0's self-attention (the precomputed candidate rows)
  const float* q0 = low ? low[0].Wq_s : w->Wq_s;
  const float* k0 = low ? low[0].Wk_s : w->Wk_s;
  const float* v0 = low ? low[0].Wv_s : w->Wv_s;
  const float* o0 = low ? low[0].Wo_s : w->Wo_s;
  s->pre_ln1_g = low ? low[0].ln1_g : w->ln1_g;
  s->pre_ln1_b = low ? low[0].ln1_b : w->ln1_b;
  const int r1 = 2 * nd;  // row blocks of h in Wcat1
  float *Wcat1 = nullptr, *Wcat2 = nullptr;
  cudaError_t e = cudaMalloc(&Wcat1, (size_t)r1 * h * D * sizeof(float));
  if (e == cudaSuccess) e = cudaMalloc(&Wcat2, (size_t)3 * h * h * sizeof(float));
  if (e == cudaSuccess) e = cudaMalloc(&s->P1s, (size_t)r1 * h * 6 * D * sizeof(uint16_t));
  if (e == cudaSuccess) e = cudaMalloc(&s->P2s, (size_t)3 * h * 6 * h * sizeof(uint16_t));
  if (e == cudaSuccess && nd > 1) e = cudaMalloc(&s->Wf, (size_t)(nd - 1) * 3 * h * h * sizeof(float));
  if (e == cudaSuccess && nd > 1) e = cudaMalloc(&s->dec_dev, (size_t)nd * sizeof(DecLayerDev));
  const float rs = 1.0f / std::sqrt((float)h);
  if (e == cudaSuccess) e = cudaMemcpy2D(Wcat1, D * sizeof(float), w->W_in, D * sizeof(float), D * sizeof(float), h, cudaMemcpyDeviceToDevice);
  // Wq_p^T Wk_p / sqrt(h): (i, j) = sum_k Wq_p[k, i] Wk_p[k, j]
  if (e == cudaSuccess) e = fold_matmul(w->Wq_p, 1, h, w->Wk_p, D, 1, Wcat1 + (size_t)h * D, D, h, D, h, rs, 0);
  // the layers before the last: Wq_c^T Wk_c / sqrt(h) and Wo_c Wv_c
  for (int l = 0; e == cudaSuccess && l + 1 < nd; ++l) {
    e = fold_matmul(low[l].Wq_c, 1, h, low[l].Wk_c, D, 1, Wcat1 + (size_t)(2 + 2 * l) * h * D, D, h, D, h, rs, 0);
    if (e == cudaSuccess)
      e = fold_matmul(low[l].Wo_c, h, 1, low[l].Wv_c, D, 1, Wcat1 + (size_t)(3 + 2 * l) * h * D, D, h, D, h, 1.f, 0);
  }
  // Wq / sqrt(h), as Wq times the identity through the same fold kernel
  std::vector<float> eye;
  float* dI = nullptr;
  if (e == cudaSuccess) {
    eye.assign((size_t)h * h, 0.f);
    for (int i = 0; i < h; ++i) eye[(size_t)i * h + i] = 1.f;
    e = cudaMalloc(&dI, (size_t)h * h * sizeof(float));
    if (e == cudaSuccess) e = cudaMemcpy(dI, eye.data(), eye.size() * sizeof(float), cudaMemcpyHostToDevice);
  }
  // [Wq / sqrt(h); Wk; Wo Wv] of one self-attention into dst [3h, h]
  auto fold_self = [&](const float* Wq, const float* Wk, const float* Wv, const float* Wo, float* dst) {
    cudaError_t r = fold_matmul(Wq, h, 1, dI, h, 1, dst, h, h, h, h, rs, 0);
    if (r == cudaSuccess) r = cudaMemcpy(dst + (size_t)h * h, Wk, (size_t)h * h * sizeof(float), cudaMemcpyDeviceToDevice);
    // Wo Wv: (i, j) = sum_k Wo[i, k] Wv[k, j]
    if (r == cudaSuccess) r = fold_matmul(Wo, h, 1, Wv, h, 1, dst + (size_t)2 * h * h, h, h, h, h, 1.f, 0);
    return r;
  };
  if (e == cudaSuccess) e = fold_self(q0, k0, v0, o0, Wcat2);
  std::vector<DecLayerDev> dd(nd);
  for (int l = 0; e == cudaSuccess && l < nd; ++l) {
    DecLayerDev& L = dd[l];
    memset(&L, 0, sizeof(L));
    const bool last = l == nd - 1;
    if (l >= 1) {
      L.Wf = s->Wf + (size_t)(l - 1) * 3 * h * h;
      e = last ? fold_self(w->Wq_s, w->Wk_s, w->Wv_s, w->Wo_s, const_cast<float*>(L.Wf))
               : fold_self(low[l].Wq_s, low[l].Wk_s, low[l].Wv_s, low[l].Wo_s, const_cast<float*>(L.Wf));
      L.ln1_g = last ? w->ln1_g : low[l].ln1_g;
      L.ln1_b = last ? w->ln1_b : low[l].ln1_b;
    }
    if (!last) {
      L.ln2_g = low[l].ln2_g; L.ln2_b = low[l].ln2_b;
      L.ln3_g = low[l].ln3_g; L.ln3_b = low[l].ln3_b;
      L.W1 = static_cast<const __nv_bfloat16*>(low[l].W1);
      L.W2 = static_cast<const __nv_bfloat16*>(low[l].W2);
    }
  }
  if (e == cudaSuccess && nd > 1) e = cudaMemcpy(s->dec_dev, dd.data(), nd * sizeof(DecLayerDev), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = split6_weights(Wcat1, r1 * h, D, s->P1s, 0);
  if (e == cudaSuccess) e = split6_weights(Wcat2, 3 * h, h, s->P2s, 0);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (dI) cudaFree(dI);
  if (Wcat1) cudaFree(Wcat1);
  if (Wcat2) cudaFree(Wcat2);
  if (e != cudaSuccess) {
    sp_selector_destroy(s);
    return cuda_fail(e, "sp_selector_create (fold)");
  }
  std::string msg;
  bool ok = make_gemm_b(&s->P1, s->P1s, r1 * h, 6 * D, &msg) && make_gemm_b(&s->P2, s->P2s, 3 * h, 6 * h, &msg);
  if (ok && c.n_enc_layers > 0) {
    ok = make_gemm_b(&s->Wp, w->W_p, D, c.D_text, &msg);
    for (int i = 0; ok && i < c.n_enc_layers; ++i) {
      ok = make_gemm_b(&s->enc_qkv[i], w->enc_wqkv[i], 3 * D, D, &msg) &&
           make_gemm_b(&s->enc_o[i], w->enc_wo[i], D, D, &msg) &&
           make_gemm_b(&s->enc_1[i], w->enc_w1[i], c.enc_ffn, D, &msg) &&
           make_gemm_b(&s->enc_2[i], w->enc_w2[i], D, c.enc_ffn, &msg);
    }
  }
  if (!ok) {
    sp_selector_destroy(s);
    return fail(SP_ERR_CUDA, "sp_selector_create: %s", msg.c_str());
  }
  *out = s;
  return SP_OK;
}

void sp_selector_destroy(sp_selector* s) {
  if (!s) return;
  if (s->P1s) cudaFree(s->P1s);
  if (s->P2s) cudaFree(s->P2s);
  if (s->Wf) cudaFree(s->Wf);
  if (s->dec_dev) cudaFree(s->dec_dev);
  delete s;
}

namespace {

struct SelPlan {
  BatchDesc bd;
  int E = 0, nvis = 0, ntxt = 0, T_enc = 0, max_enc = 0, rows = 0, k_max = 0;
  bool encoder = false;
};

sp_status plan_select(const sp_selector* s, const sp_select_in* in, SelPlan* p) {
  if (!s || !in) return fail(SP_ERR_INVALID_ARG, "sp_select: NULL selector or input");
  std::string msg;
  if (!fill_batch_desc(&p->bd, in->B, in->n_vis, in->n_txt, in->group_size, &msg))
    return fail(SP_ERR_SHAPE, "sp_select: %s", msg.c_str());
  if (in->g < 1 || in->g > 16) return fail(SP_ERR_SHAPE, "g must be in 1..16");
  if (in->k_max < 1 || in->k_max > SP_MAX_KMAX) return fail(SP_ERR_SHAPE, "k_max must be in 1..SP_MAX_KMAX");
  p->E = p->bd.ep_off[in->B];
  p->k_max = in->k_max;
  p->nvis = p->bd.vis_off[in->B];
  p->ntxt = p->bd.txt_off[in->B];
  p->rows = p->nvis + 2;
  p->encoder = (in->H == nullptr);
  p->T_enc = p->nvis + p->ntxt;
  p->max_enc = 0;
  for (int b = 0; b < in->B; ++b) p->max_enc = std::max(p->max_enc, in->n_vis[b] + in->n_txt[b]);
  return SP_OK;
}

size_t select_ws(const sp_selector* s, const SelPlan& p, const sp_select_out* out, Carve& cv,
                 void** parts) {
  const int D = s->cfg.D, h = s->cfg.h, F = s->cfg.enc_ffn;
  float *P = nullptr, *R = nullptr, *Mall, *ZK, *XL, *QKVs;
  void *Abf = nullptr, *QKV = nullptr, *O = nullptr, *F1 = nullptr;
  int* enc_cu = nullptr;
  void* gsk = nullptr;  // stream-K scratch of the encoder GEMMs (the precompute GEMMs run whole tiles)
  if (p.encoder && s->cfg.n_enc_layers > 0) {
    gsk = cv.take<char>(gemm_scratch_bytes());
    P = cv.take<float>((size_t)std::max(p.ntxt, 1) * D);
    R = cv.take<float>((size_t)p.T_enc * D);
    Abf = cv.take<uint16_t>((size_t)p.T_enc * D);
    QKV = cv.take<uint16_t>((size_t)p.T_enc * 3 * D);
    O = cv.take<uint16_t>((size_t)p.T_enc * D);
    F1 = cv.take<uint16_t>((size_t)p.T_enc * F);
    enc_cu = cv.take<int>(SP_MAX_BATCH + 1);
  } else if (p.encoder) {
    R = cv.take<float>((size_t)p.T_enc * D);
  }
  Mall = cv.take<float>((size_t)p.rows * D);
  ZK = cv.take<float>((size_t)p.rows * 2 * s->n_dec * h);
  XL = cv.take<float>((size_t)p.rows * h);
  QKVs = cv.take<float>((size_t)p.rows * 3 * h);
  void* Asp = cv.take<uint16_t>((size_t)p.rows * 3 * std::max(D, h));  // split operand of the precompute GEMMs
  int* order = (out && out->order) ? nullptr : cv.take<int>((size_t)p.E * SP_MAX_KMAX);
  int* epc = (out && out->ep_count) ? nullptr : cv.take<int>((size_t)p.E);
  // self-attention rows of decoder layers >= 1, per episode and history position
  float* dcache = s->n_dec > 1 ? cv.take<float>((size_t)p.E * (s->n_dec - 1) * (p.k_max + 1) * 2 * h) : nullptr;
  if (parts) {
    parts[0] = P; parts[1] = R; parts[2] = Abf; parts[3] = QKV; parts[4] = O; parts[5] = F1;
    parts[6] = enc_cu; parts[7] = Mall; parts[8] = ZK; parts[9] = XL; parts[10] = QKVs;
    parts[11] = order; parts[12] = epc; parts[13] = gsk; parts[14] = Asp; parts[15] = dcache;
  }
  return cv.off;
}

// Runs the encoder stack (Eq. 3) on X / E_text into R (fp32 residual rows).
sp_status run_encoder(const sp_selector* s, const sp_select_in* in, const SelPlan& p, void** parts,
                      int* err, cudaStream_t st) {
  const sp_selector_cfg& c = s->cfg;
  const int D = c.D;
  float* P = (float*)parts[0];
  float* R = (float*)parts[1];
  void* Abf = parts[2];
  void* QKV = parts[3];
  void* O = parts[4];
  void* F1 = parts[5];
  int* enc_cu = (int*)parts[6];
  const GemmScratch gs = gemm_scratch_at(parts[13]);  // cleared by the caller
  std::string msg;
  if (p.ntxt > 0) {
    CUtensorMap tE;
    if (!encode_tmap_bf16(&tE, in->E_text, p.ntxt, c.D_text, 128, &msg)) return fail(SP_ERR_CUDA, "%s", msg.c_str());
    GemmEpi ep;
    ep.kind = EPI_F32;
    ep.out = P;
    ep.ldo = D;
    SP_CUDA(gemm_bf16(tE, p.ntxt, nullptr, s->Wp, D, ep, err, st, &gs), "text projection");
  }
  SP_CUDA(assemble_encoder_input(p.bd, in->X, P, D, s->w.ln_text_g, s->w.ln_text_b, c.ln_eps, c.g_text, R,
                                 p.T_enc, st), "encoder input");
  SP_CUDA(write_enc_cu(p.bd, enc_cu, st), "encoder offsets");
  CUtensorMap tA, tO, tF;
  if (!encode_tmap_bf16(&tA, Abf, p.T_enc, D, 128, &msg) || !encode_tmap_bf16(&tO, O, p.T_enc, D, 128, &msg) ||
      !encode_tmap_bf16(&tF, F1, p.T_enc, c.enc_ffn, 128, &msg))
    return fail(SP_ERR_CUDA, "%s", msg.c_str());
  const int nh = D / c.enc_head_dim;
  for (int l = 0; l < c.n_enc_layers; ++l) {
    SP_CUDA(layernorm_f32(R, D, s->w.enc_ln1_g[l], s->w.enc_ln1_b[l], nullptr, Abf, D, p.T_enc, D, c.ln_eps, 1.f, st), "enc ln1");
    GemmEpi e1;
    e1.kind = EPI_BF16;
    e1.out = QKV;
    e1.ldo = 3 * D;
    SP_CUDA(gemm_bf16(tA, p.T_enc, nullptr, s->enc_qkv[l], 3 * D, e1, err, st, &gs), "enc qkv");
    SP_CUDA(attention_varlen(QKV, O, enc_cu, in->B, p.max_enc, p.T_enc, nh, nh, c.enc_head_dim, false,
                             gs.attn_sched, err, st),
            "enc attention");
    GemmEpi e2;
    e2.kind = EPI_F32_ACC;
    e2.out = R;
    e2.ldo = D;
    SP_CUDA(gemm_bf16(tO, p.T_enc, nullptr, s->enc_o[l], D, e2, err, st, &gs), "enc o");
    SP_CUDA(layernorm_f32(R, D, s->w.enc_ln2_g[l], s->w.enc_ln2_b[l], nullptr, Abf, D, p.T_enc, D, c.ln_eps, 1.f, st), "enc ln2");
    GemmEpi e3;
    e3.kind = EPI_GELU_BF16;
    e3.out = F1;
    e3.ldo = c.enc_ffn;
    SP_CUDA(gemm_bf16(tA, p.T_enc, nullptr, s->enc_1[l], c.enc_ffn, e3, err, st, &gs), "enc fc1");
    SP_CUDA(gemm_bf16(tF, p.T_enc, nullptr, s->enc_2[l], D, e2, err, st, &gs), "enc fc2");
  }
  return SP_OK;
}

}  // namespace

size_t sp_select_workspace(const sp_selector* s, const sp_select_in* in) {
  SelPlan p;
  if (plan_select(s, in, &p) != SP_OK) return 0;
  Carve cv(nullptr);
  return select_ws(s, p, nullptr, cv, nullptr) + 256;
}

static sp_status select_impl(const sp_selector* s, const sp_select_in* in, const sp_select_out* out, void* ws,
                             size_t ws_bytes, cudaStream_t st, const sp_train_args* tr = nullptr) {
  SelPlan p;
  sp_status rs = plan_select(s, in, &p);
  if (rs != SP_OK) return rs;
  if (s->n_dec > 1 && (in->g != 1 || tr))
    return fail(SP_ERR_UNSUPPORTED, "sp_select: a decoder of %d layers takes g = 1 (and no training aggregates)",
                s->n_dec);
  if (tr) {
    if (!tr->score || !tr->kbar || (reinterpret_cast<uintptr_t>(tr->score) & 3) ||
        (reinterpret_cast<uintptr_t>(tr->kbar) & 3))
      return fail(SP_ERR_INVALID_ARG, "sp_select_train: score and kbar (4-byte aligned) are required");
    if (!(tr->tau > 0.f) || !std::isfinite(tr->tau) || !(tr->beta > 0.f) || !(tr->beta <= 1.f))
      return fail(SP_ERR_INVALID_ARG, "sp_select_train: need tau > 0 and beta in (0, 1]");
    if (in->g != 1) return fail(SP_ERR_UNSUPPORTED, "sp_select_train: the rollout of Eqs. 5-7 takes g = 1");
    bool ks = true;
    size_t sm = 0;
    select_cluster_size(p.bd, s->cfg.h, in->k_max, &ks, &sm);
    if (!ks) return fail(SP_ERR_UNSUPPORTED, "sp_select_train: an episode's keys must fit shared memory");
  }
  if (!out || !out->idx || !out->count) return fail(SP_ERR_INVALID_ARG, "sp_select: idx and count are required");
  if (!in->stop_bias) return fail(SP_ERR_INVALID_ARG, "sp_select: stop_bias is required");
  if (p.encoder && (!in->X || (p.ntxt > 0 && s->cfg.n_enc_layers > 0 && !in->E_text)))
    return fail(SP_ERR_INVALID_ARG, "sp_select: X / E_text required when H is NULL");
  if ((in->X && !al16(in->X)) || (in->E_text && !al16(in->E_text)) || (in->H && !al16(in->H)))
    return fail(SP_ERR_ALIGN, "sp_select: inputs must be 16-byte aligned");
  int need_cap = 0;
  for (int b = 0; b < in->B; ++b) {
    const int n = in->n_vis[b], gs = in->group_size > 0 ? in->group_size : n;
    int c = 0;
    for (int s0 = 0; s0 < n; s0 += gs) c += std::min(in->k_max, std::min(gs, n - s0));
    need_cap = std::max(need_cap, c);
  }
  if (out->k_cap < need_cap) return fail(SP_ERR_SHAPE, "sp_select: k_cap %d < largest possible count %d", out->k_cap, need_cap);
  Carve cv(ws);
  void* parts[16];
  const size_t need = select_ws(s, p, out, cv, parts) + 256;
  if (!ws || ws_bytes < need) return fail(SP_ERR_WORKSPACE, "sp_select: workspace %zu < %zu bytes", ws_bytes, need);
  if (!al16(ws)) return fail(SP_ERR_ALIGN, "sp_select: workspace must be 16-byte aligned");
  int* err = out->err;
  const int D = s->cfg.D, h = s->cfg.h;
  const GemmScratch gs = gemm_scratch_at(parts[13]);
  SP_CUDA(gemm_scratch_clear(gs, st), "GEMM scratch");

  if (p.encoder && s->cfg.n_enc_layers > 0) {
    rs = run_encoder(s, in, p, parts, err, st);
    if (rs != SP_OK) return rs;
    SP_CUDA(gather_memory(p.bd, (float*)parts[1], nullptr, s->w.s_stop, s->w.s_start, (float*)parts[7], D, st), "memory");
  } else if (p.encoder) {
    // no encoder blocks: H = X (converted to fp32)
    SP_CUDA(bf16_to_f32(in->X, (float*)parts[1], p.nvis, nullptr, D, st), "X to fp32");
    BatchDesc flat = p.bd;
    for (int b = 0; b <= in->B; ++b) flat.txt_off[b] = 0;
    SP_CUDA(gather_memory(flat, (float*)parts[1], nullptr, s->w.s_stop, s->w.s_start, (float*)parts[7], D, st), "memory");
  } else {
    SP_CUDA(gather_memory(p.bd, nullptr, in->H, s->w.s_stop, s->w.s_start, (float*)parts[7], D, st), "memory");
  }
  float* Mall = (float*)parts[7];
  if (out->memory)
    SP_CUDA(cudaMemcpyAsync(out->memory, Mall, (size_t)p.nvis * D * sizeof(float), cudaMemcpyDeviceToDevice, st),
            "memory copy");
  float* ZK = (float*)parts[8];
  float* XL = (float*)parts[9];
  float* QKVs = (float*)parts[10];
  // candidate precompute (fp32): [z | KT] = M [W_in; Wq_p^T Wk_p / sqrt h]^T, x = LN1(z),
  // [QS | KS | VT] = x [Wq_s / sqrt h; Wk_s; Wo_s Wv_s]^T
  // (fp32-accurate products on the bf16 tensor cores: three-way operand split)
  {
    void* Asp = parts[14];
    std::string msg;
    CUtensorMap t1, t2;
    if (!encode_tmap_bf16(&t1, Asp, p.rows, 3 * D, 128, &msg) || !encode_tmap_bf16(&t2, Asp, p.rows, 3 * h, 128, &msg))
      return fail(SP_ERR_CUDA, "%s", msg.c_str());
    GemmEpi e1;
    e1.kind = EPI_F32;
    e1.out = ZK;
    e1.ldo = 2 * s->n_dec * h;
    const GemmASplit a1 = split3_a_map(D), a2 = split3_a_map(h);
    SP_CUDA(split3_bf16(Mall, D, p.rows, D, Asp, st), "precompute split 1");
    SP_CUDA(gemm_bf16(t1, p.rows, nullptr, s->P1, 2 * s->n_dec * h, e1, err, st, nullptr, &a1), "precompute 1");
    SP_CUDA(layernorm_f32(ZK, 2 * s->n_dec * h, s->pre_ln1_g, s->pre_ln1_b, XL, nullptr, h, p.rows, h, s->cfg.ln_eps,
                          1.f, st), "ln1");
    GemmEpi e2;
    e2.kind = EPI_F32;
    e2.out = QKVs;
    e2.ldo = 3 * h;
    SP_CUDA(split3_bf16(XL, h, p.rows, h, Asp, st), "precompute split 2");
    SP_CUDA(gemm_bf16(t2, p.rows, nullptr, s->P2, 3 * h, e2, err, st, nullptr, &a2), "precompute 2");
  }

  SelectArgs a;
  a.Z = ZK; a.ldz = 2 * s->n_dec * h;
  a.KT = ZK + h; a.ldkt = 2 * s->n_dec * h;
  a.QS = QKVs; a.ldqs = 3 * h;
  a.KS = QKVs + h; a.ldks = 3 * h;
  a.VT = QKVs + 2 * h; a.ldvt = 3 * h;
  a.ln2_g = s->w.ln2_g; a.ln2_b = s->w.ln2_b;
  a.ln_eps = s->cfg.ln_eps;
  a.stop_row = p.nvis;
  a.start_row = p.nvis + 1;
  a.stop_bias = in->stop_bias;
  a.h = h; a.k_max = in->k_max; a.g = in->g;
  a.order = out->order ? out->order : (int*)parts[11];
  a.ep_count = out->ep_count ? out->ep_count : (int*)parts[12];
  a.margin = out->margin; a.gap = out->gap; a.rounds = out->rounds;
  a.err = err;
  a.score = tr ? tr->score : nullptr;
  a.kbar = tr ? tr->kbar : nullptr;
  a.inv_tau = tr ? 1.f / tr->tau : 1.f;
  a.beta = tr ? tr->beta : 1.f;
  a.n_dec = s->n_dec;
  a.dec = s->dec_dev;
  a.KC = ZK + 2 * h;
  a.dcache = static_cast<float*>(parts[15]);
  a.dcache_ep = (size_t)(s->n_dec - 1) * (in->k_max + 1) * 2 * h;
  bool keys_smem = true;
  size_t smem = 0;
  const int C = select_cluster_size(p.bd, h, in->k_max, &keys_smem, &smem, s->n_dec > 1);
  SP_CUDA(select_launch(p.bd, p.E, a, C, keys_smem, smem, st), "selection");
  SP_CUDA(restore_launch(p.bd, a.order, a.ep_count, in->k_max, out->idx, out->k_cap, out->count, err, st), "restore");
  return SP_OK;
}

sp_status sp_select(const sp_selector* s, const sp_select_in* in, const sp_select_out* out, void* ws,
                    size_t ws_bytes, sp_stream stream) {
  return select_impl(s, in, out, ws, ws_bytes, (cudaStream_t)stream);
}

sp_status sp_select_train(const sp_selector* s, const sp_select_in* in, const sp_select_out* out,
                          const sp_train_args* train, void* ws, size_t ws_bytes, sp_stream stream) {
  if (!train) return fail(SP_ERR_INVALID_ARG, "sp_select_train: train arguments are required");
  return select_impl(s, in, out, ws, ws_bytes, (cudaStream_t)stream, train);
}

sp_status sp_soft_topk(int B, const int* n_vis, int group_size, const float* score, const float* kbar, float tau,
                       float* alpha, float* k_out, sp_stream stream) {
  if (B < 1 || B > SP_MAX_BATCH || !n_vis) return fail(SP_ERR_INVALID_ARG, "sp_soft_topk: bad batch");
  if (!score || !kbar || !alpha) return fail(SP_ERR_INVALID_ARG, "sp_soft_topk: score, kbar and alpha are required");
  if (!(tau > 0.f) || !std::isfinite(tau)) return fail(SP_ERR_INVALID_ARG, "sp_soft_topk: need tau > 0");
  std::vector<int> zeros(B, 0);
  BatchDesc bd;
  std::string msg;
  if (!fill_batch_desc(&bd, B, n_vis, zeros.data(), group_size, &msg))
    return fail(SP_ERR_SHAPE, "sp_soft_topk: %s", msg.c_str());
  SP_CUDA(soft_topk_launch(bd, bd.ep_off[B], score, kbar, tau, alpha, k_out, (cudaStream_t)stream), "soft top-k");
  return SP_OK;
}

sp_status sp_vp_gate(int rows, int D, const void* X, const void* noise, const float* alpha, void* out,
                     sp_stream stream) {
  if (rows < 0 || D <= 0 || D % 8) return fail(SP_ERR_SHAPE, "sp_vp_gate: rows >= 0 and D a multiple of 8");
  if (rows == 0) return SP_OK;
  if (!X || !noise || !alpha || !out) return fail(SP_ERR_INVALID_ARG, "sp_vp_gate: NULL pointer");
  if (!al16(X) || !al16(noise) || !al16(out)) return fail(SP_ERR_ALIGN, "sp_vp_gate: X, noise, out 16-byte aligned");
  SP_CUDA(vp_gate_launch(X, noise, alpha, out, rows, D, (cudaStream_t)stream), "vp gate");
  return SP_OK;
}

}  // extern "C"

namespace sp {
sp_status report(sp_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

sp_status select_with_workspace(const sp_selector* s, const sp_select_in* in, const sp_select_out* out, void* ws,
                                size_t ws_bytes, cudaStream_t st) {
  return select_impl(s, in, out, ws, ws_bytes, st);
}
}  // namespace sp

extern "C" {

// ------------------------------------------------------------------ compaction

static sp_status compact_impl(const sp_compact_in* in, const sp_compact_out* out, cudaStream_t st) {
  if (!in || !out) return fail(SP_ERR_INVALID_ARG, "sp_compact: NULL argument");
  BatchDesc bd;
  std::string msg;
  if (!fill_batch_desc(&bd, in->B, in->n_vis, in->n_txt, 0, &msg)) return fail(SP_ERR_SHAPE, "sp_compact: %s", msg.c_str());
  if (!in->X || !in->idx || !in->count || !out->packed || !out->cu_seqlens || !out->pos)
    return fail(SP_ERR_INVALID_ARG, "sp_compact: X, idx, count, packed, cu_seqlens, pos are required");
  if (bd.txt_off[in->B] > 0 && !in->text) return fail(SP_ERR_INVALID_ARG, "sp_compact: text is required");
  if (in->W_vis <= 0 || in->W_vis % 8 || in->W_txt <= 0 || in->W_txt % 8)
    return fail(SP_ERR_SHAPE, "sp_compact: W_vis and W_txt must be positive multiples of 8");
  if (in->k_cap < 0) return fail(SP_ERR_SHAPE, "sp_compact: k_cap must be >= 0");
  const bool index_mode = out->vis_src != nullptr;
  if (index_mode && out->vis_packed) return fail(SP_ERR_INVALID_ARG, "sp_compact: vis_src and vis_packed are exclusive");
  const bool direct = out->vis_packed == nullptr && !index_mode;
  if (direct && in->W_vis != in->W_txt) return fail(SP_ERR_SHAPE, "sp_compact: direct mode needs W_vis == W_txt");
  if (!direct && (!out->vis_row_map || !out->vis_cu))
    return fail(SP_ERR_INVALID_ARG, "sp_compact: vis_row_map and vis_cu required with vis_packed / vis_src");
  if (!al16(in->X) || (in->text && !al16(in->text)) || !al16(out->packed) || (out->vis_packed && !al16(out->vis_packed)))
    return fail(SP_ERR_ALIGN, "sp_compact: row buffers must be 16-byte aligned");
  const int T_cap = sp_packed_cap(in->B, in->n_vis, in->n_txt, in->k_cap);
  SP_CUDA(compact_launch(bd, in->X, in->W_vis, in->text, in->W_txt, in->idx, in->k_cap, in->count, out->packed,
                         out->cu_seqlens, out->pos, out->vis_packed, out->vis_row_map, out->vis_cu, out->vis_src,
                         T_cap, out->err, st),
          "compaction");
  return SP_OK;
}

sp_status sp_compact(const sp_compact_in* in, const sp_compact_out* out, sp_stream stream) {
  return compact_impl(in, out, (cudaStream_t)stream);
}

// ------------------------------------------------------------------ model

sp_status sp_model_create(const sp_model_cfg* cfg, const sp_model_weights* w, sp_model** out) {
  if (!cfg || !w || !out) return fail(SP_ERR_INVALID_ARG, "sp_model_create: NULL argument");
  *out = nullptr;
  sp_status st = check_device();
  if (st != SP_OK) return st;
  const sp_model_cfg c = *cfg;
  if (c.n_layers < 1 || c.n_layers > SP_MAX_LM_LAYERS) return fail(SP_ERR_SHAPE, "n_layers out of range");
  if (c.d <= 0 || c.d % 128) return fail(SP_ERR_SHAPE, "d must be a multiple of 128");
  if (c.head_dim != 64 && c.head_dim != 128) return fail(SP_ERR_SHAPE, "head_dim must be 64 or 128");
  if (c.n_heads < 1 || c.n_kv_heads < 1 || c.n_heads % c.n_kv_heads) return fail(SP_ERR_SHAPE, "n_kv_heads must divide n_heads");
  const int qkv = (c.n_heads + 2 * c.n_kv_heads) * c.head_dim;
  if (qkv % 256) return fail(SP_ERR_SHAPE, "(n_heads + 2 n_kv_heads) head_dim must be a multiple of 256");
  if ((c.n_heads * c.head_dim) % 128) return fail(SP_ERR_SHAPE, "n_heads head_dim must be a multiple of 128");
  if (c.ffn <= 0 || c.ffn % 128) return fail(SP_ERR_SHAPE, "ffn must be a multiple of 128");
  if (c.max_pos < 1 || c.max_pos > (1 << 20)) return fail(SP_ERR_SHAPE, "max_pos out of range");
  if (!(c.rope_theta > 0.f) || !(c.rms_eps > 0.f)) return fail(SP_ERR_INVALID_ARG, "rope_theta and rms_eps must be > 0");
  if (c.proj_kind < SP_PROJ_NONE || c.proj_kind > SP_PROJ_MLP2_GELU) return fail(SP_ERR_INVALID_ARG, "bad proj_kind");
  {
    const int* ms = c.mrope_section;
    const int sum = ms[0] + ms[1] + ms[2];
    if (sum != 0 && (ms[0] < 0 || ms[1] < 0 || ms[2] < 0 || (ms[0] | ms[1] | ms[2]) & 1 || sum != c.head_dim / 2))
      return fail(SP_ERR_SHAPE, "mrope_section: three even pair counts summing to head_dim / 2 (or all zero)");
  }
  if (c.proj_kind != SP_PROJ_NONE) {
    if (c.proj_in <= 0 || c.proj_in % 64) return fail(SP_ERR_SHAPE, "proj_in must be a multiple of 64");
    if (!w->proj_w1) return fail(SP_ERR_INVALID_ARG, "proj_w1 required");
    if (c.proj_kind == SP_PROJ_MLP2_GELU) {
      if (c.proj_hidden <= 0 || c.proj_hidden % 128) return fail(SP_ERR_SHAPE, "proj_hidden must be a multiple of 128");
      if (!w->proj_w2) return fail(SP_ERR_INVALID_ARG, "proj_w2 required");
    }
  }
  for (int l = 0; l < c.n_layers; ++l)
    if (!w->wqkv[l] || !w->wo[l] || !w->wgu[l] || !w->wdown[l]) return fail(SP_ERR_INVALID_ARG, "layer %d weights missing", l);

  sp_model* m = new (std::nothrow) sp_model_s();
  if (!m) return fail(SP_ERR_INVALID_ARG, "out of host memory");
  m->cfg = c;
  m->w = *w;
  // rotary table: angle = pos * theta^(-2i/dh), in double, stored as fp32 (cos, sin)
  const int half = c.head_dim / 2;
  std::vector<float2> tab((size_t)c.max_pos * half);
  for (int p = 0; p < c.max_pos; ++p)
    for (int i = 0; i < half; ++i) {
      const double inv = std::pow((double)c.rope_theta, -(2.0 * i) / (double)c.head_dim);
      const double ang = (double)p * inv;
      tab[(size_t)p * half + i] = make_float2((float)std::cos(ang), (float)std::sin(ang));
    }
  cudaError_t e = cudaMalloc(&m->rope, tab.size() * sizeof(float2));
  if (e == cudaSuccess) e = cudaMemcpy(m->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) {
    sp_model_destroy(m);
    return cuda_fail(e, "sp_model_create (rope table)");
  }
  std::string msg;
  bool ok = true;
  m->qkv.resize(c.n_layers);
  m->o.resize(c.n_layers);
  m->gu.resize(c.n_layers);
  m->down.resize(c.n_layers);
  for (int l = 0; ok && l < c.n_layers; ++l) {
    ok = make_gemm_b(&m->qkv[l], w->wqkv[l], qkv, c.d, &msg) &&
         make_gemm_b(&m->o[l], w->wo[l], c.d, c.n_heads * c.head_dim, &msg) &&
         make_gemm_b(&m->gu[l], w->wgu[l], 2 * c.ffn, c.d, &msg) &&
         make_gemm_b(&m->down[l], w->wdown[l], c.d, c.ffn, &msg);
  }
  if (ok && c.proj_kind == SP_PROJ_LINEAR) ok = make_gemm_b(&m->p1, w->proj_w1, c.d, c.proj_in, &msg);
  if (ok && c.proj_kind == SP_PROJ_MLP2_GELU)
    ok = make_gemm_b(&m->p1, w->proj_w1, c.proj_hidden, c.proj_in, &msg) &&
         make_gemm_b(&m->p2, w->proj_w2, c.d, c.proj_hidden, &msg);
  if (!ok) {
    sp_model_destroy(m);
    return fail(SP_ERR_CUDA, "sp_model_create: %s", msg.c_str());
  }
  *out = m;
  return SP_OK;
}

void sp_model_destroy(sp_model* m) {
  if (!m) return;
  if (m->rope) cudaFree(m->rope);
  delete m;
}

// ------------------------------------------------------------------ projector

static size_t project_ws(const sp_model* m, int rows_cap, Carve& cv, void** tmp, void** gsk = nullptr,
                         float** splitk = nullptr, size_t* splitk_floats = nullptr) {
  void* t = nullptr;
  if (m->cfg.proj_kind == SP_PROJ_MLP2_GELU) t = cv.take<uint16_t>((size_t)std::max(rows_cap, 1) * m->cfg.proj_hidden);
  void* g = m->cfg.proj_kind != SP_PROJ_NONE ? cv.take<char>(gemm_scratch_bytes()) : nullptr;
  float* sk = nullptr;
  size_t skf = 0;
  if (m->cfg.proj_kind != SP_PROJ_NONE && rows_cap <= 128) {
    skf = gemm_splitk_floats(std::max(m->cfg.proj_hidden, m->cfg.d));
    sk = cv.take<float>(skf);
  }
  if (tmp) *tmp = t;
  if (gsk) *gsk = g;
  if (splitk) *splitk = sk;
  if (splitk_floats) *splitk_floats = skf;
  return cv.off;
}

size_t sp_project_workspace(const sp_model* m, int rows_cap) {
  if (!m || rows_cap < 0) return 0;
  Carve cv(nullptr);
  return project_ws(m, rows_cap, cv, nullptr) + 256;
}

static sp_status project_impl(const sp_model* m, const sp_project_io* io, void* ws, size_t ws_bytes, cudaStream_t st) {
  if (!m || !io) return fail(SP_ERR_INVALID_ARG, "sp_project: NULL argument");
  const sp_model_cfg& c = m->cfg;
  if (c.proj_kind == SP_PROJ_NONE) return SP_OK;
  if (io->B < 1 || io->B > SP_MAX_BATCH || io->rows_cap < 0) return fail(SP_ERR_SHAPE, "sp_project: bad B / rows_cap");
  const bool gather = io->vis_src != nullptr;
  if ((!gather && !io->vis_packed) || !io->vis_row_map || !io->vis_cu || !io->packed)
    return fail(SP_ERR_INVALID_ARG, "sp_project: vis_packed (or vis_src), vis_row_map, vis_cu and packed are required");
  if (gather && (!io->X || io->rows_X < 1)) return fail(SP_ERR_INVALID_ARG, "sp_project: vis_src needs X and rows_X >= 1");
  if ((!gather && !al16(io->vis_packed)) || (gather && !al16(io->X)) || !al16(io->packed))
    return fail(SP_ERR_ALIGN, "sp_project: buffers must be 16-byte aligned");
  if (io->rows_cap == 0) return SP_OK;
  Carve cv(ws);
  void* tmp = nullptr;
  void* gsk = nullptr;
  float* spk = nullptr;
  size_t spkf = 0;
  const size_t need = project_ws(m, io->rows_cap, cv, &tmp, &gsk, &spk, &spkf) + 256;
  const bool have_ws = ws && ws_bytes >= need;
  if (c.proj_kind == SP_PROJ_MLP2_GELU && !have_ws)
    return fail(SP_ERR_WORKSPACE, "sp_project: workspace %zu < %zu bytes", ws_bytes, need);
  // a linear projector runs without a workspace too (whole GEMM tiles only)
  GemmScratch gs = gemm_scratch_at(have_ws ? gsk : nullptr);
  if (have_ws) {
    gs.splitk = spk;
    gs.splitk_floats = spkf;
  }
  SP_CUDA(gemm_scratch_clear(gs, st), "GEMM scratch");
  std::string msg;
  // the first GEMM's A: the packed kept rows, or the rows of X they come from
  // (row-gather map: a box of one row, gathered four rows per copy)
  CUtensorMap tV;
  if (gather ? !encode_tmap_bf16(&tV, io->X, io->rows_X, c.proj_in, 1, &msg)
             : !encode_tmap_bf16(&tV, io->vis_packed, io->rows_cap, c.proj_in, 128, &msg))
    return fail(SP_ERR_CUDA, "%s", msg.c_str());
  const int* a_rows = gather ? io->vis_src : nullptr;
  const int* M_dev = io->vis_cu + io->B;
  GemmEpi sc;
  sc.kind = EPI_SCATTER_BF16;
  sc.out = io->packed;
  sc.ldo = c.d;
  sc.row_map = io->vis_row_map;
  if (c.proj_kind == SP_PROJ_LINEAR) {
    SP_CUDA(gemm_bf16(tV, io->rows_cap, M_dev, m->p1, c.d, sc, io->err, st, &gs, nullptr, nullptr, a_rows),
            "projector");
    return SP_OK;
  }
  GemmEpi g1;
  g1.kind = EPI_GELU_BF16;
  g1.out = tmp;
  g1.ldo = c.proj_hidden;
  SP_CUDA(gemm_bf16(tV, io->rows_cap, M_dev, m->p1, c.proj_hidden, g1, io->err, st, &gs, nullptr, nullptr, a_rows),
          "projector fc1");
  CUtensorMap tT;
  if (!encode_tmap_bf16(&tT, tmp, io->rows_cap, c.proj_hidden, 128, &msg)) return fail(SP_ERR_CUDA, "%s", msg.c_str());
  SP_CUDA(gemm_bf16(tT, io->rows_cap, M_dev, m->p2, c.d, sc, io->err, st, &gs), "projector fc2");
  return SP_OK;
}

sp_status sp_project(const sp_model* m, const sp_project_io* io, void* ws, size_t ws_bytes, sp_stream stream) {
  return project_impl(m, io, ws, ws_bytes, (cudaStream_t)stream);
}

// ------------------------------------------------------------------ prefill

struct PrefillParts {
  float* h32;
  void *xb, *qkv, *ob, *act, *gsk;
  float2* mrows = nullptr;  // mRoPE: per packed row (cos, sin) of every rotation pair
  int* mident = nullptr;    // mRoPE: row r -> r
  float* splitk = nullptr;  // small-M split-K planes (T_cap <= 128)
  size_t splitk_floats = 0;
  float* dattn = nullptr;   // decode: attention partials of the key ranges
  int* dcnt = nullptr;      // decode: per layer, per (sequence, kv head) range counters
};

constexpr int kDecodeSplits = 16;  // key ranges per sequence in a generation step, at most

static size_t model_max_n(const sp_model_cfg& c) {
  return (size_t)std::max(std::max((c.n_heads + 2 * c.n_kv_heads) * c.head_dim, c.d), 2 * c.ffn);
}

static size_t prefill_ws(const sp_model* m, int T_cap, bool own_residual, Carve& cv, PrefillParts* p) {
  const sp_model_cfg& c = m->cfg;
  const size_t T = (size_t)std::max(T_cap, 1);
  PrefillParts q;
  q.h32 = own_residual ? cv.take<float>(T * c.d) : nullptr;
  q.xb = cv.take<uint16_t>(T * c.d);
  q.qkv = cv.take<uint16_t>(T * (c.n_heads + 2 * c.n_kv_heads) * c.head_dim);
  q.ob = cv.take<uint16_t>(T * c.n_heads * c.head_dim);
  q.act = cv.take<uint16_t>(T * c.ffn);
  q.gsk = cv.take<char>(gemm_scratch_bytes());
  if (c.mrope_section[0] + c.mrope_section[1] + c.mrope_section[2] > 0) {
    q.mrows = cv.take<float2>(T * (c.head_dim / 2));
    q.mident = cv.take<int>(T);
  }
  if (T_cap <= 128) {
    q.splitk_floats = gemm_splitk_floats((int)model_max_n(c));
    q.splitk = cv.take<float>(q.splitk_floats);
  }
  if (p) *p = q;
  return cv.off;
}

size_t sp_prefill_workspace(const sp_model* m, int T_cap, int max_seqlen_cap) {
  if (!m || T_cap < 0 || max_seqlen_cap < 0) return 0;
  Carve cv(nullptr);
  return prefill_ws(m, T_cap, true, cv, nullptr) + 256;
}

static sp_status prefill_impl(const sp_model* m, const sp_prefill_io* io, void* ws, size_t ws_bytes, cudaStream_t st) {
  if (!m || !io) return fail(SP_ERR_INVALID_ARG, "sp_prefill: NULL argument");
  const sp_model_cfg& c = m->cfg;
  if (io->B < 1 || io->B > SP_MAX_BATCH || io->T_cap < 0 || io->max_seqlen_cap < 0)
    return fail(SP_ERR_SHAPE, "sp_prefill: bad B / T_cap / max_seqlen_cap");
  const bool mrope = c.mrope_section[0] + c.mrope_section[1] + c.mrope_section[2] > 0;
  if (!mrope && io->max_seqlen_cap > c.max_pos)  // (mRoPE positions are checked on the device)
    return fail(SP_ERR_SHAPE, "sp_prefill: max_seqlen_cap %d > max_pos %d", io->max_seqlen_cap, c.max_pos);
  if (!io->x || !io->cu_seqlens || !io->pos || !io->hidden) return fail(SP_ERR_INVALID_ARG, "sp_prefill: x, cu_seqlens, pos, hidden required");
  if (!al16(io->x) || !al16(io->hidden) || (io->residual && !al16(io->residual)) || (io->kv && !al16(io->kv)))
    return fail(SP_ERR_ALIGN, "sp_prefill: buffers must be 16-byte aligned");
  if (io->kv && io->kv_S_cap < io->max_seqlen_cap)
    return fail(SP_ERR_SHAPE, "sp_prefill: kv_S_cap %d < max_seqlen_cap %d", io->kv_S_cap, io->max_seqlen_cap);
  if (mrope && (!io->pos3 || !al16(io->pos3)))
    return fail(SP_ERR_INVALID_ARG, "sp_prefill: an mRoPE model needs pos3 (16-byte aligned)");
  if (io->T_cap == 0) return SP_OK;
  Carve cv(ws);
  PrefillParts p;
  const size_t need = prefill_ws(m, io->T_cap, io->residual == nullptr, cv, &p) + 256;
  if (!ws || ws_bytes < need) return fail(SP_ERR_WORKSPACE, "sp_prefill: workspace %zu < %zu bytes", ws_bytes, need);
  if (!al16(ws)) return fail(SP_ERR_ALIGN, "sp_prefill: workspace must be 16-byte aligned");
  float* h32 = io->residual ? io->residual : p.h32;
  const int T_cap = io->T_cap;
  const int* T_dev = io->cu_seqlens + io->B;
  const int dq = c.n_heads * c.head_dim, qkvw = (c.n_heads + 2 * c.n_kv_heads) * c.head_dim;
  std::string msg;
  CUtensorMap tX, tO, tA;
  if (!encode_tmap_bf16(&tX, p.xb, T_cap, c.d, 128, &msg) || !encode_tmap_bf16(&tO, p.ob, T_cap, dq, 128, &msg) ||
      !encode_tmap_bf16(&tA, p.act, T_cap, c.ffn, 128, &msg))
    return fail(SP_ERR_CUDA, "%s", msg.c_str());
  GemmScratch gs = gemm_scratch_at(p.gsk);
  gs.splitk = p.splitk;
  gs.splitk_floats = p.splitk_floats;
  SP_CUDA(gemm_scratch_clear(gs, st), "GEMM scratch");
  SP_CUDA(bf16_to_f32(io->x, h32, T_cap, T_dev, c.d, st), "embed");
  // the attention's last key block reads up to 127 rows past the packed length
  // (weighted by zero); keep them finite: the QKV GEMMs leave them untouched
  SP_CUDA(zero_rows_after(p.qkv, (size_t)qkvw * 2, T_dev, T_cap, 128, st), "qkv tail");
  if (mrope)
    SP_CUDA(mrope_rows_launch(m->rope, c.max_pos, c.head_dim / 2, io->pos3, c.mrope_section[0],
                              c.mrope_section[0] + c.mrope_section[1], T_dev, T_cap, p.mrows, p.mident, io->err, st),
            "mrope rows");
  for (int l = 0; l < c.n_layers; ++l) {
    SP_CUDA(rmsnorm_f32_to_bf16(h32, m->w.attn_norm[l], p.xb, T_cap, T_dev, c.d, c.rms_eps, st), "attn norm");
    GemmEpi eq;
    eq.kind = EPI_BF16_ROPE;
    eq.out = p.qkv;
    eq.ldo = qkvw;
    eq.rope = mrope ? p.mrows : m->rope;
    eq.pos = mrope ? p.mident : io->pos;
    eq.max_pos = mrope ? T_cap : c.max_pos;
    eq.head_dim = c.head_dim;
    eq.rope_cols = (c.n_heads + c.n_kv_heads) * c.head_dim;
    SP_CUDA(gemm_bf16(tX, T_cap, T_dev, m->qkv[l], qkvw, eq, io->err, st, &gs), "qkv");
    if (io->kv) {
      void* kv_l = static_cast<uint16_t*>(io->kv) + (size_t)l * 2 * io->B * io->kv_S_cap * c.n_kv_heads * c.head_dim;
      SP_CUDA(kv_store(p.qkv, io->cu_seqlens, io->pos, io->B, T_cap, c.n_heads, c.n_kv_heads, c.head_dim, kv_l,
                       io->kv_S_cap, io->err, st), "kv cache");
    }
    SP_CUDA(attention_varlen(p.qkv, p.ob, io->cu_seqlens, io->B, io->max_seqlen_cap, T_cap, c.n_heads, c.n_kv_heads,
                             c.head_dim, true, gs.attn_sched, io->err, st), "attention");
    GemmEpi er;
    er.kind = EPI_F32_ACC;
    er.out = h32;
    er.ldo = c.d;
    SP_CUDA(gemm_bf16(tO, T_cap, T_dev, m->o[l], c.d, er, io->err, st, &gs), "o");
    SP_CUDA(rmsnorm_f32_to_bf16(h32, m->w.mlp_norm[l], p.xb, T_cap, T_dev, c.d, c.rms_eps, st), "mlp norm");
    GemmEpi eg;
    eg.kind = EPI_SWIGLU_BF16;
    eg.out = p.act;
    eg.ldo = c.ffn;
    eg.up_off = c.ffn;
    SP_CUDA(gemm_bf16(tX, T_cap, T_dev, m->gu[l], 2 * c.ffn, eg, io->err, st, &gs), "gate/up");
    SP_CUDA(gemm_bf16(tA, T_cap, T_dev, m->down[l], c.d, er, io->err, st, &gs), "down");
  }
  SP_CUDA(rmsnorm_f32_to_f32(h32, m->w.final_norm, io->hidden, T_cap, T_dev, c.d, c.rms_eps, st), "final norm");
  return SP_OK;
}

sp_status sp_prefill(const sp_model* m, const sp_prefill_io* io, void* ws, size_t ws_bytes, sp_stream stream) {
  return prefill_impl(m, io, ws, ws_bytes, (cudaStream_t)stream);
}

sp_status sp_mrope_positions(int B, const int* n_vis, const int* n_txt, const int* grid_w, const int* idx, int k_cap,
                             const int* count, int* pos3, int T_cap, int* err, sp_stream stream) {
  BatchDesc bd;
  std::string msg;
  if (!fill_batch_desc(&bd, B, n_vis, n_txt, 0, &msg)) return fail(SP_ERR_SHAPE, "sp_mrope_positions: %s", msg.c_str());
  if (!grid_w || !idx || !count || !pos3) return fail(SP_ERR_INVALID_ARG, "sp_mrope_positions: NULL argument");
  if (k_cap < 1 || T_cap < 0) return fail(SP_ERR_SHAPE, "sp_mrope_positions: bad k_cap / T_cap");
  if (!al16(pos3)) return fail(SP_ERR_ALIGN, "sp_mrope_positions: pos3 must be 16-byte aligned");
  GridDesc gd;
  for (int b = 0; b < B; ++b) {
    if (grid_w[b] < 1 || grid_w[b] > n_vis[b]) return fail(SP_ERR_SHAPE, "sp_mrope_positions: grid_w[%d] out of 1..N_b", b);
    gd.grid_w[b] = grid_w[b];
  }
  SP_CUDA(mrope_positions_launch(bd, gd, idx, k_cap, count, pos3, T_cap, err, (cudaStream_t)stream), "mrope positions");
  return SP_OK;
}

// ------------------------------------------------------------------ decode

static size_t decode_ws(const sp_model* m, int B, Carve& cv, PrefillParts* p) {
  // the prefill's buffers at B rows (the single-CTA GEMM path: no stream-K scratch)
  const sp_model_cfg& c = m->cfg;
  const size_t R = (size_t)std::max(B, 1);
  PrefillParts q;
  q.h32 = cv.take<float>(R * c.d);
  q.xb = cv.take<uint16_t>(R * c.d);
  q.qkv = cv.take<uint16_t>(R * (c.n_heads + 2 * c.n_kv_heads) * c.head_dim);
  q.ob = cv.take<uint16_t>(R * c.n_heads * c.head_dim);
  q.act = cv.take<uint16_t>(R * c.ffn);
  q.gsk = nullptr;
  if (B <= 128) {
    q.splitk_floats = gemm_splitk_floats((int)model_max_n(c));
    q.splitk = cv.take<float>(q.splitk_floats);
  }
  q.dattn = cv.take<float>(decode_attention_floats((int)R, c.n_heads, c.head_dim, kDecodeSplits));
  q.dcnt = cv.take<int>((size_t)c.n_layers * R * c.n_kv_heads);
  if (p) *p = q;
  return cv.off;
}

size_t sp_decode_workspace(const sp_model* m, int B) {
  if (!m || B < 1) return 0;
  Carve cv(nullptr);
  return decode_ws(m, B, cv, nullptr) + 256;
}

static sp_status decode_impl(const sp_model* m, const sp_decode_io* io, void* ws, size_t ws_bytes, cudaStream_t st) {
  if (!m || !io) return fail(SP_ERR_INVALID_ARG, "sp_decode: NULL argument");
  const sp_model_cfg& c = m->cfg;
  if (io->B < 1 || io->B > SP_MAX_BATCH || io->kv_S_cap < 1 || io->max_len_cap < 1 || io->max_len_cap > io->kv_S_cap)
    return fail(SP_ERR_SHAPE, "sp_decode: bad B / kv_S_cap / max_len_cap");
  if (!io->rope_pos && io->max_len_cap > c.max_pos)  // (explicit rotary positions are checked on the device)
    return fail(SP_ERR_SHAPE, "sp_decode: max_len_cap %d > max_pos %d", io->max_len_cap, c.max_pos);
  if (!io->x || !io->lens || !io->kv || !io->hidden) return fail(SP_ERR_INVALID_ARG, "sp_decode: x, lens, kv, hidden required");
  if (c.n_heads / c.n_kv_heads > 8)
    return fail(SP_ERR_UNSUPPORTED, "sp_decode: more than 8 query heads per key / value head");
  if (!al16(io->x) || !al16(io->kv) || !al16(io->hidden)) return fail(SP_ERR_ALIGN, "sp_decode: buffers must be 16-byte aligned");
  Carve cv(ws);
  PrefillParts p;
  const size_t need = decode_ws(m, io->B, cv, &p) + 256;
  if (!ws || ws_bytes < need) return fail(SP_ERR_WORKSPACE, "sp_decode: workspace %zu < %zu bytes", ws_bytes, need);
  if (!al16(ws)) return fail(SP_ERR_ALIGN, "sp_decode: workspace must be 16-byte aligned");
  const int B = io->B;
  const int dq = c.n_heads * c.head_dim, qkvw = (c.n_heads + 2 * c.n_kv_heads) * c.head_dim;
  const size_t layer_elems = (size_t)2 * B * io->kv_S_cap * c.n_kv_heads * c.head_dim;
  std::string msg;
  CUtensorMap tX, tO, tA, tX16, tO16, tA16;  // box rows 128 / 16 (weight-streaming GEMMs)
  if (!encode_tmap_bf16(&tX, p.xb, B, c.d, 128, &msg) || !encode_tmap_bf16(&tO, p.ob, B, dq, 128, &msg) ||
      !encode_tmap_bf16(&tA, p.act, B, c.ffn, 128, &msg) || !encode_tmap_bf16(&tX16, p.xb, B, c.d, 16, &msg) ||
      !encode_tmap_bf16(&tO16, p.ob, B, dq, 16, &msg) || !encode_tmap_bf16(&tA16, p.act, B, c.ffn, 16, &msg))
    return fail(SP_ERR_CUDA, "%s", msg.c_str());
  GemmScratch gs;
  gs.splitk = p.splitk;
  gs.splitk_floats = p.splitk_floats;
  SP_CUDA(cudaMemsetAsync(p.dcnt, 0, sizeof(int) * (size_t)c.n_layers * B * c.n_kv_heads, st), "decode counters");
  SP_CUDA(bf16_to_f32(io->x, p.h32, B, nullptr, c.d, st), "embed");
  for (int l = 0; l < c.n_layers; ++l) {
    void* kv_l = static_cast<uint16_t*>(io->kv) + (size_t)l * layer_elems;
    SP_CUDA(rmsnorm_f32_to_bf16(p.h32, m->w.attn_norm[l], p.xb, B, nullptr, c.d, c.rms_eps, st), "attn norm");
    GemmEpi eq;
    eq.kind = EPI_BF16_ROPE;
    eq.out = p.qkv;
    eq.ldo = qkvw;
    eq.rope = m->rope;
    eq.pos = io->rope_pos ? io->rope_pos : io->lens;  // default: the cached length
    eq.max_pos = c.max_pos;
    eq.head_dim = c.head_dim;
    eq.rope_cols = (c.n_heads + c.n_kv_heads) * c.head_dim;
    SP_CUDA(gemm_bf16(tX, B, nullptr, m->qkv[l], qkvw, eq, io->err, st, &gs, nullptr, &tX16), "qkv");
    SP_CUDA(decode_attention(p.qkv, kv_l, io->kv_S_cap, io->lens, B, c.n_heads, c.n_kv_heads, c.head_dim,
                             io->max_len_cap, p.dattn, kDecodeSplits, p.dcnt + (size_t)l * B * c.n_kv_heads, p.ob,
                             io->err, st),
            "decode attention");
    GemmEpi er;
    er.kind = EPI_F32_ACC;
    er.out = p.h32;
    er.ldo = c.d;
    SP_CUDA(gemm_bf16(tO, B, nullptr, m->o[l], c.d, er, io->err, st, &gs, nullptr, &tO16), "o");
    SP_CUDA(rmsnorm_f32_to_bf16(p.h32, m->w.mlp_norm[l], p.xb, B, nullptr, c.d, c.rms_eps, st), "mlp norm");
    GemmEpi eg;
    eg.kind = EPI_SWIGLU_BF16;
    eg.out = p.act;
    eg.ldo = c.ffn;
    eg.up_off = c.ffn;
    SP_CUDA(gemm_bf16(tX, B, nullptr, m->gu[l], 2 * c.ffn, eg, io->err, st, &gs, nullptr, &tX16), "gate/up");
    SP_CUDA(gemm_bf16(tA, B, nullptr, m->down[l], c.d, er, io->err, st, &gs, nullptr, &tA16), "down");
  }
  SP_CUDA(rmsnorm_f32_to_f32(p.h32, m->w.final_norm, io->hidden, B, nullptr, c.d, c.rms_eps, st), "final norm");
  SP_CUDA(lens_increment(io->lens, io->rope_pos, B, io->kv_S_cap, st), "lens");
  return SP_OK;
}

sp_status sp_decode(const sp_model* m, const sp_decode_io* io, void* ws, size_t ws_bytes, sp_stream stream) {
  return decode_impl(m, io, ws, ws_bytes, (cudaStream_t)stream);
}

// ------------------------------------------------------------------ pipeline

namespace {
struct PipePlan {
  int T_cap = 0, max_len = 0, rows_cap = 0;
};

sp_status plan_pipe(const sp_selector* s, const sp_model* m, const sp_select_in& sel, int k_cap, PipePlan* p) {
  if (!s || !m) return fail(SP_ERR_INVALID_ARG, "sp_pipeline: NULL handle");
  if (sel.B < 1 || sel.B > SP_MAX_BATCH || !sel.n_vis || !sel.n_txt) return fail(SP_ERR_SHAPE, "sp_pipeline: bad batch");
  if (s->cfg.D_text != m->cfg.d) return fail(SP_ERR_SHAPE, "sp_pipeline: D_text must equal the LM width d");
  if (m->cfg.proj_kind == SP_PROJ_NONE ? s->cfg.D != m->cfg.d : s->cfg.D != m->cfg.proj_in)
    return fail(SP_ERR_SHAPE, "sp_pipeline: visual width does not match the projector input");
  p->T_cap = sp_packed_cap(sel.B, sel.n_vis, sel.n_txt, k_cap);
  if (p->T_cap < 0) return fail(SP_ERR_SHAPE, "sp_pipeline: bad sizes");
  p->max_len = 0;
  p->rows_cap = 0;
  for (int b = 0; b < sel.B; ++b) {
    p->max_len = std::max(p->max_len, std::min(sel.n_vis[b], k_cap) + sel.n_txt[b]);
    p->rows_cap += std::min(sel.n_vis[b], k_cap);
  }
  if (p->max_len > m->cfg.max_pos) return fail(SP_ERR_SHAPE, "sp_pipeline: a sequence can exceed max_pos");
  return SP_OK;
}

struct PipeParts {
  void* packed;
  int* pos;
  int* vis_src;  // the projector gathers the kept rows from X (compaction's index mode)
  int* vis_row_map;
  int* vis_cu;
  void* scratch;
  size_t scratch_bytes;
};

size_t pipe_ws(const sp_selector* s, const sp_model* m, const sp_select_in& sel, const PipePlan& pp, Carve& cv,
               PipeParts* out) {
  PipeParts q;
  q.packed = cv.take<uint16_t>((size_t)std::max(pp.T_cap, 1) * m->cfg.d);
  q.pos = cv.take<int>((size_t)std::max(pp.T_cap, 1));
  const bool proj = m->cfg.proj_kind != SP_PROJ_NONE;
  q.vis_src = proj ? cv.take<int>((size_t)std::max(pp.rows_cap, 1)) : nullptr;
  q.vis_row_map = proj ? cv.take<int>((size_t)std::max(pp.rows_cap, 1)) : nullptr;
  q.vis_cu = proj ? cv.take<int>(SP_MAX_BATCH + 1) : nullptr;
  SelPlan sp_;
  sp_select_in si = sel;
  si.H = nullptr;
  plan_select(s, &si, &sp_);
  Carve c1(nullptr), c2(nullptr), c3(nullptr);
  sp_select_out so = {};
  so.order = nullptr;
  so.ep_count = nullptr;
  const size_t a = select_ws(s, sp_, &so, c1, nullptr);
  const size_t b = project_ws(m, pp.rows_cap, c2, nullptr);
  const size_t c = prefill_ws(m, pp.T_cap, true, c3, nullptr);
  q.scratch_bytes = std::max(a, std::max(b, c)) + 256;
  q.scratch = cv.take<char>(q.scratch_bytes);
  if (out) *out = q;
  return cv.off;
}
}  // namespace

size_t sp_pipeline_workspace(const sp_selector* s, const sp_model* m, const sp_pipeline_io* io) {
  if (!io) return 0;
  PipePlan pp;
  if (plan_pipe(s, m, io->sel, io->k_cap, &pp) != SP_OK) return 0;
  SelPlan tmp;
  sp_select_in si = io->sel;
  si.H = nullptr;
  if (plan_select(s, &si, &tmp) != SP_OK) return 0;
  Carve cv(nullptr);
  return pipe_ws(s, m, io->sel, pp, cv, nullptr) + 256;
}

static sp_status pipeline_impl(const sp_selector* s, const sp_model* m, const sp_pipeline_io* io, void* ws,
                               size_t ws_bytes, cudaStream_t st) {
  if (!io) return fail(SP_ERR_INVALID_ARG, "sp_pipeline: NULL io");
  PipePlan pp;
  sp_status r = plan_pipe(s, m, io->sel, io->k_cap, &pp);
  if (r != SP_OK) return r;
  if (!io->idx || !io->count || !io->cu_seqlens || !io->hidden) return fail(SP_ERR_INVALID_ARG, "sp_pipeline: idx, count, cu_seqlens, hidden required");
  Carve cv(ws);
  PipeParts q;
  const size_t need = pipe_ws(s, m, io->sel, pp, cv, &q) + 256;
  if (!ws || ws_bytes < need) return fail(SP_ERR_WORKSPACE, "sp_pipeline: workspace %zu < %zu bytes", ws_bytes, need);
  if (!al16(ws)) return fail(SP_ERR_ALIGN, "sp_pipeline: workspace must be 16-byte aligned");

  sp_select_in si = io->sel;
  si.H = nullptr;
  sp_select_out so = {};
  so.idx = io->idx;
  so.k_cap = io->k_cap;
  so.count = io->count;
  so.err = io->err;
  r = select_impl(s, &si, &so, q.scratch, q.scratch_bytes, st);
  if (r != SP_OK) return r;

  const bool proj = m->cfg.proj_kind != SP_PROJ_NONE;
  sp_compact_in ci = {};
  ci.B = si.B;
  ci.n_vis = si.n_vis;
  ci.n_txt = si.n_txt;
  ci.X = si.X;
  ci.W_vis = s->cfg.D;
  ci.text = si.E_text;
  ci.W_txt = m->cfg.d;
  ci.idx = io->idx;
  ci.k_cap = io->k_cap;
  ci.count = io->count;
  sp_compact_out co = {};
  co.packed = q.packed;
  co.cu_seqlens = io->cu_seqlens;
  co.pos = q.pos;
  co.vis_src = q.vis_src;
  co.vis_row_map = q.vis_row_map;
  co.vis_cu = q.vis_cu;
  co.err = io->err;
  r = compact_impl(&ci, &co, st);
  if (r != SP_OK) return r;
  if (proj) {
    int rows_X = 0;
    for (int b = 0; b < si.B; ++b) rows_X += si.n_vis[b];
    sp_project_io pj = {};
    pj.B = si.B;
    pj.rows_cap = pp.rows_cap;
    pj.vis_row_map = q.vis_row_map;
    pj.vis_cu = q.vis_cu;
    pj.packed = q.packed;
    pj.err = io->err;
    pj.X = si.X;
    pj.rows_X = std::max(1, rows_X);
    pj.vis_src = q.vis_src;
    r = project_impl(m, &pj, q.scratch, q.scratch_bytes, st);
    if (r != SP_OK) return r;
  }
  sp_prefill_io pf = {};
  pf.B = si.B;
  pf.T_cap = pp.T_cap;
  pf.max_seqlen_cap = pp.max_len;
  pf.x = q.packed;
  pf.cu_seqlens = io->cu_seqlens;
  pf.pos = q.pos;
  pf.hidden = io->hidden;
  pf.residual = nullptr;
  pf.err = io->err;
  return prefill_impl(m, &pf, q.scratch, q.scratch_bytes, st);
}

sp_status sp_pipeline(const sp_selector* s, const sp_model* m, const sp_pipeline_io* io, void* ws, size_t ws_bytes,
                      sp_stream stream) {
  return pipeline_impl(s, m, io, ws, ws_bytes, (cudaStream_t)stream);
}

// ------------------------------------------------------------------ pipeline from host buffers

namespace {
struct HostParts {
  void* X;
  void* E;
  float* bias;
  int* idx;
  int* count;
  int* cu;
  float* hidden;
  int* err;
  void* inner;
};

size_t host_ws(const sp_selector* s, const sp_model* m, const sp_pipeline_host_io* io, const PipePlan& pp, Carve& cv,
               HostParts* out, size_t* inner_bytes) {
  const sp_select_in& sel = io->sel;
  int nvis = 0, ntxt = 0;
  for (int b = 0; b < sel.B; ++b) { nvis += sel.n_vis[b]; ntxt += sel.n_txt[b]; }
  const int E = sp_num_episodes(sel.B, sel.n_vis, sel.group_size);
  HostParts q;
  q.X = cv.take<uint16_t>((size_t)nvis * s->cfg.D);
  q.E = cv.take<uint16_t>((size_t)std::max(ntxt, 1) * s->cfg.D_text);
  q.bias = cv.take<float>((size_t)std::max(E, 1));
  q.idx = cv.take<int>((size_t)sel.B * io->k_cap);
  q.count = cv.take<int>(sel.B);
  q.cu = cv.take<int>(sel.B + 1);
  q.hidden = cv.take<float>((size_t)std::max(pp.T_cap, 1) * m->cfg.d);
  q.err = cv.take<int>(4);
  Carve c2(nullptr);
  const size_t ib = pipe_ws(s, m, sel, pp, c2, nullptr) + 256;
  q.inner = cv.take<char>(ib);
  if (out) *out = q;
  if (inner_bytes) *inner_bytes = ib;
  return cv.off;
}
}  // namespace

size_t sp_pipeline_host_workspace(const sp_selector* s, const sp_model* m, const sp_pipeline_host_io* io) {
  if (!io) return 0;
  PipePlan pp;
  if (plan_pipe(s, m, io->sel, io->k_cap, &pp) != SP_OK) return 0;
  if (sp_num_episodes(io->sel.B, io->sel.n_vis, io->sel.group_size) < 0) return 0;
  Carve cv(nullptr);
  return host_ws(s, m, io, pp, cv, nullptr, nullptr) + 256;
}

sp_status sp_pipeline_host(const sp_selector* s, const sp_model* m, const sp_pipeline_host_io* io, void* ws,
                           size_t ws_bytes, sp_stream stream) {
  cudaStream_t st = (cudaStream_t)stream;
  if (!io) return fail(SP_ERR_INVALID_ARG, "sp_pipeline_host: NULL io");
  PipePlan pp;
  sp_status r = plan_pipe(s, m, io->sel, io->k_cap, &pp);
  if (r != SP_OK) return r;
  const sp_select_in& sel = io->sel;
  if (!sel.X || !sel.stop_bias || !io->host_idx || !io->host_count || !io->host_cu_seqlens || !io->host_hidden)
    return fail(SP_ERR_INVALID_ARG, "sp_pipeline_host: host buffers missing");
  const int E = sp_num_episodes(sel.B, sel.n_vis, sel.group_size);
  if (E < 0) return fail(SP_ERR_SHAPE, "sp_pipeline_host: bad batch");
  Carve cv(ws);
  HostParts q;
  size_t inner = 0;
  const size_t need = host_ws(s, m, io, pp, cv, &q, &inner) + 256;
  if (!ws || ws_bytes < need) return fail(SP_ERR_WORKSPACE, "sp_pipeline_host: workspace %zu < %zu bytes", ws_bytes, need);
  int nvis = 0, ntxt = 0;
  for (int b = 0; b < sel.B; ++b) { nvis += sel.n_vis[b]; ntxt += sel.n_txt[b]; }
  SP_CUDA(cudaMemcpyAsync(q.X, sel.X, (size_t)nvis * s->cfg.D * 2, cudaMemcpyHostToDevice, st), "copy X");
  if (ntxt > 0) SP_CUDA(cudaMemcpyAsync(q.E, sel.E_text, (size_t)ntxt * s->cfg.D_text * 2, cudaMemcpyHostToDevice, st), "copy E");
  SP_CUDA(cudaMemcpyAsync(q.bias, sel.stop_bias, (size_t)E * 4, cudaMemcpyHostToDevice, st), "copy stop_bias");
  SP_CUDA(cudaMemsetAsync(q.err, 0, 16, st), "clear error word");
  sp_pipeline_io dio = {};
  dio.sel = sel;
  dio.sel.X = q.X;
  dio.sel.E_text = q.E;
  dio.sel.stop_bias = q.bias;
  dio.sel.H = nullptr;
  dio.k_cap = io->k_cap;
  dio.idx = q.idx;
  dio.count = q.count;
  dio.cu_seqlens = q.cu;
  dio.hidden = q.hidden;
  dio.err = q.err;
  r = pipeline_impl(s, m, &dio, q.inner, inner, st);
  if (r != SP_OK) return r;
  SP_CUDA(cudaMemcpyAsync(io->host_idx, q.idx, (size_t)sel.B * io->k_cap * 4, cudaMemcpyDeviceToHost, st), "copy idx");
  SP_CUDA(cudaMemcpyAsync(io->host_count, q.count, (size_t)sel.B * 4, cudaMemcpyDeviceToHost, st), "copy count");
  SP_CUDA(cudaMemcpyAsync(io->host_cu_seqlens, q.cu, (size_t)(sel.B + 1) * 4, cudaMemcpyDeviceToHost, st), "copy cu");
  SP_CUDA(cudaMemcpyAsync(io->host_hidden, q.hidden, (size_t)pp.T_cap * m->cfg.d * 4, cudaMemcpyDeviceToHost, st), "copy hidden");
  return SP_OK;
}

// ------------------------------------------------------------------ profiling

sp_status sp_profile_begin(int capacity) {
  for (cudaEvent_t e : g_prof.ev) cudaEventDestroy(e);
  g_prof = Prof();
  if (capacity <= 0) return SP_OK;
  g_prof.ev.resize((size_t)2 * capacity);
  for (auto& e : g_prof.ev) SP_CUDA(cudaEventCreate(&e), "cudaEventCreate");
  g_prof.kind.assign(capacity, 0);
  g_prof.flops.assign(capacity, 0.0);
  g_prof.bytes.assign(capacity, 0.0);
  g_prof.cap = capacity;
  g_prof.n = 0;
  g_prof.on = true;
  return SP_OK;
}

sp_status sp_profile_end(double* ms, long long* launches, double* flops, double* bytes) {
  if (!g_prof.on) return fail(SP_ERR_INVALID_ARG, "sp_profile_end: profiling is not active");
  for (int k = 0; k < SP_K_COUNT; ++k) {
    if (ms) ms[k] = 0.0;
    if (launches) launches[k] = 0;
    if (flops) flops[k] = 0.0;
    if (bytes) bytes[k] = 0.0;
  }
  sp_status st = SP_OK;
  if (g_prof.n > 0) {
    cudaError_t e = cudaEventSynchronize(g_prof.ev[2 * g_prof.n - 1]);
    if (e != cudaSuccess) st = cuda_fail(e, "sp_profile_end");
  }
  for (int i = 0; st == SP_OK && i < g_prof.n; ++i) {
    float t = 0.f;
    cudaEventElapsedTime(&t, g_prof.ev[2 * i], g_prof.ev[2 * i + 1]);
    const int k = g_prof.kind[i];
    if (ms) ms[k] += t;
    if (launches) launches[k] += 1;
    if (flops) flops[k] += g_prof.flops[i];
    if (bytes) bytes[k] += g_prof.bytes[i];
  }
  for (cudaEvent_t e : g_prof.ev) cudaEventDestroy(e);
  g_prof = Prof();
  return st;
}

}  // extern "C"
