// Host-side interfaces between the translation units of libstepprune.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "stepprune.h"

namespace sp {

// Per-image offsets known on the host, passed to kernels by value.
struct BatchDesc {
  int B;
  int group_size;                 // candidates per episode (resolved: > 0 only when grouping)
  int vis_off[SP_MAX_BATCH + 1];  // prefix of n_vis
  int txt_off[SP_MAX_BATCH + 1];  // prefix of n_txt
  int ep_off[SP_MAX_BATCH + 1];   // prefix of episodes per image
};

// grid width (tokens per row) of every image of a batch (mRoPE positions)
struct GridDesc {
  int grid_w[SP_MAX_BATCH];
};

// Launch with programmatic stream serialization (the kernel must call
// pdl_wait before touching memory other kernels use); off when the
// environment sets SP_PDL=0.
bool pdl_enabled();
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

bool fill_batch_desc(BatchDesc* d, int B, const int* n_vis, const int* n_txt, int group_size,
                     std::string* msg);

int device_sm_count();

// ------------------------------------------------------------- profiling
void prof_begin_launch(cudaStream_t st);
void prof_end_launch(cudaStream_t st, int kind, double flops, double bytes);
bool prof_enabled();

// ------------------------------------------------------------- tensor maps
bool encode_tmap_bf16(CUtensorMap* map, const void* ptr, uint64_t rows, uint64_t cols,
                      uint32_t box_rows, std::string* msg);
// 2-D map over a row-major [rows, cols] matrix of 2- or 4-byte elements with a
// box of box_cols x box_rows and 128-byte swizzle (box_cols * esize <= 128).
bool encode_tmap_2d(CUtensorMap* map, const void* ptr, bool f32, uint64_t rows, uint64_t cols,
                    uint32_t box_cols, uint32_t box_rows, std::string* msg);

// ------------------------------------------------------------- tcgen05 GEMM
enum EpiKind {
  EPI_BF16 = 0,         // out bf16 = acc
  EPI_BF16_ROPE = 1,    // out bf16 = acc with rotate-half RoPE on columns < rope_cols
  EPI_F32 = 2,          // out fp32 = acc
  EPI_F32_ACC = 3,      // out fp32 += acc (residual add)
  EPI_GELU_BF16 = 4,    // out bf16 = gelu(acc)
  EPI_SWIGLU_BF16 = 5,  // out bf16 [.., N/2] = silu(gate) * up
  EPI_SCATTER_BF16 = 6  // out bf16 row row_map[r] = acc
};

struct GemmEpi {
  int kind = EPI_BF16;
  void* out = nullptr;
  int ldo = 0;                       // elements
  const int* row_map = nullptr;      // EPI_SCATTER_BF16
  const float2* rope = nullptr;      // [max_pos, head_dim / 2] (cos, sin)
  const int* pos = nullptr;          // [rows]
  int max_pos = 0;
  int head_dim = 0;
  int rope_cols = 0;
  int up_off = 0;                    // EPI_SWIGLU_BF16: row of B where the 'up' half starts
};

// Weight operand: the B tensor maps for both tile widths.
struct GemmB {
  CUtensorMap map128;  // box rows 64  (BN = 128 -> two boxes of 64)
  CUtensorMap map256;  // box rows 128 (BN = 256 -> two boxes of 128)
  int N = 0;           // rows of B
  int K = 0;
};

bool make_gemm_b(GemmB* b, const void* w, int N, int K, std::string* msg);
int gemm_pair_policy(int M_cap, int N_acc, int kind);

// C[M, N] = A[M, K] B[N, K]^T with the given epilogue.  A's tensor map has box
// rows 128.  M_dev (device int, may be NULL) bounds the rows actually computed;
// M_cap bounds it on the host.  N_out is the accumulator width (N of B, or the
// tile columns for SWIGLU: 2 F).
// Scratch of the CTA-pair GEMM's stream-K tail: per SM pair one fp32 256 x 256
// partial tile and 8 ready flags, then the attention's two scheduling counters.
// The flags and counters must be zero when a kernel starts; every launch
// leaves them zero, so one gemm_scratch_clear per API call does.
// Without scratch (NULL) the GEMM runs whole tiles only.
struct GemmScratch {
  float* part = nullptr;
  int* flags = nullptr;
  int slots = 0;
  int* attn_sched = nullptr;  // the attention's ticket counter (two ints after the flags)
  float* splitk = nullptr;   // small-M split-K partial planes (NULL: no split)
  size_t splitk_floats = 0;
};
size_t gemm_scratch_bytes();
// fp32 scratch that lets small-M GEMMs (M <= 128) of width <= max_n_acc split K.
size_t gemm_splitk_floats(int max_n_acc);
GemmScratch gemm_scratch_at(void* p);  // p: gemm_scratch_bytes() bytes, 256-byte aligned (or NULL)
cudaError_t gemm_scratch_clear(const GemmScratch& g, cudaStream_t st);

// K-segment map of the A operand: A's k-coordinate k (of the GEMM's K = B.K)
// lies in segment s = k / seg and is read from column ((map >> 4s) & 15) * seg
// + k % seg of A's tensor map (seg = 0: identity).  Lets one stored copy of a
// part feed several K segments (the split fp32 product, precompute.cu).
struct GemmASplit {
  int seg = 0;
  uint32_t map = 0;
};

// The weight-streaming GEMM without an epilogue (M_cap <= 32 rows): fp32
// partial planes [ks][N_acc][32] (plane row n = output column n, column m =
// row m of A) in sk.splitk, *ks_out ranges, to be summed in range order by the
// consumer.  cudaErrorNotSupported when the shape or scratch does not allow it.
cudaError_t gemm_swap_partials(const CUtensorMap& A16, int M_cap, const GemmB& B, int N_acc, int* err,
                               cudaStream_t st, const GemmScratch& sk, int* ks_out);

// A16 (optional): A's tensor map with box rows 16.  With it, M_cap <= 32 and
// split-K scratch, the GEMM streams the weights as the MMA's 128-row operand
// (generation steps); the result and epilogue are the same.
// a_rows (device, may be NULL): A row r is row a_rows[r] of the tensor A's
// map describes, which then has a box of 64 columns by one row (the row-gather
// form: encode_tmap_bf16 with box_rows 1): the gather of Algorithm 1 step 5
// folded into the operand load (single-CTA and CTA-pair kernels; not the
// weight-streaming form).
cudaError_t gemm_bf16(const CUtensorMap& A, int M_cap, const int* M_dev, const GemmB& B,
                      int N_acc, const GemmEpi& e, int* err, cudaStream_t st,
                      const GemmScratch* sk = nullptr, const GemmASplit* as = nullptr,
                      const CUtensorMap* A16 = nullptr, const int* a_rows = nullptr);

// ------------------------------------------------------------- candidate precompute
// out [rows, 3K] bf16 = the three bf16 parts of x [rows, K] (fp32, row stride ldx).
cudaError_t split3_bf16(const float* x, int ldx, int rows, int K, void* out, cudaStream_t st);
// out [N, 6K] bf16 = the weight segments b0 b1 b0 b2 b1 b0 of w [N, K] (fp32).
cudaError_t split6_weights(const float* w, int N, int K, void* out, cudaStream_t st);
GemmASplit split3_a_map(int K);
cudaError_t fold_matmul(const float* A, long sai, long sak, const float* B, long sbk, long sbj,
                        float* C, int ldc, int I, int J, int K, float scale, cudaStream_t st);

// ------------------------------------------------------------- norms and small kernels
// rows from row_count (device, may be NULL) bounded by rows_cap.
cudaError_t rmsnorm_f32_to_bf16(const float* x, const float* gain, void* out, int rows_cap,
                                const int* row_count, int d, float eps, cudaStream_t st);
cudaError_t rmsnorm_f32_to_f32(const float* x, const float* gain, float* out, int rows_cap,
                               const int* row_count, int d, float eps, cudaStream_t st);
cudaError_t layernorm_f32(const float* x, int ldx, const float* gain, const float* bias, float* out_f32,
                          void* out_bf16, int ldo, int rows, int d, float eps, float scale,
                          cudaStream_t st);
// Zeroes rows [T, T + nrows) (below rows_cap) of a row-major buffer, T = *row_count.
cudaError_t zero_rows_after(void* buf, size_t row_bytes, const int* row_count, int rows_cap, int nrows,
                            cudaStream_t st);
cudaError_t bf16_to_f32(const void* x, float* out, int rows_cap, const int* row_count, int d,
                        cudaStream_t st);
cudaError_t assemble_encoder_input(const BatchDesc& bd, const void* X, const float* P, int D,
                                   const float* ln_g, const float* ln_b, float eps, float g_text,
                                   float* R, int rows, cudaStream_t st);
cudaError_t gather_memory(const BatchDesc& bd, const float* R, const float* H, const float* s_stop,
                          const float* s_start, float* Mall, int D, cudaStream_t st);
cudaError_t write_enc_cu(const BatchDesc& bd, int* cu, cudaStream_t st);

// ------------------------------------------------------------- key / value cache and decode
// Cache layout: layer block [2][B][S_cap][Hkv * dh] bf16 (K then V).
cudaError_t kv_store(const void* qkv, const int* cu, const int* pos, int B, int T_cap, int Hq, int Hkv, int dh,
                     void* kv_l, int S_cap, int* err, cudaStream_t st);
// One generation step's attention, the new key / value appended to the cache
// at lens[b] on the way: out [B, Hq dh] bf16.  Keys split into at most
// max_splits ranges per sequence; `part` holds decode_attention_floats() fp32
// partials, `cnt` B * Hkv ints that must be zero at the launch.
size_t decode_attention_floats(int B, int Hq, int dh, int max_splits);
cudaError_t decode_attention(const void* qkv, void* kv_l, int S_cap, const int* lens, int B, int Hq, int Hkv, int dh,
                             int max_len, float* part, int max_splits, int* cnt, void* out, int* err,
                             cudaStream_t st);
cudaError_t lens_increment(int* lens, int* rope_pos, int B, int S_cap, cudaStream_t st);

// ------------------------------------------------------------- attention
// Varlen attention over packed qkv [rows_cap, (Hq + 2 Hkv) dh] bf16 -> out [T, Hq dh] bf16
// (rows of sequence b from cu_seqlens[b]; rows_cap bounds the buffer for TMA).
// sched: two device ints, zero before the launch and left zero by it (the
// work-item ticket counter; GemmScratch::attn_sched), or NULL for a static
// assignment of the items to the CTAs.
cudaError_t attention_varlen(const void* qkv, void* out, const int* cu_seqlens, int B,
                             int max_seqlen_cap, int rows_cap, int Hq, int Hkv, int dh, bool causal,
                             int* sched, int* err, cudaStream_t st);

// ------------------------------------------------------------- selection
// A pointer-decoder layer's runtime weights (decoders of several layers).
// Layer 0's self-attention rows and every layer's folded cross-attention rows
// are precomputed per candidate; what depends on the history is applied here.
struct DecLayerDev {
  const float* Wf;                       // [3h, h]: [Wq_s / sqrt h; Wk_s; Wo_s Wv_s] (layers >= 1)
  const float* ln1_g; const float* ln1_b;  // (layers >= 1)
  const float* ln2_g; const float* ln2_b;  // before the cross-attention (layers before the last)
  const float* ln3_g; const float* ln3_b;  // before the FFN (layers before the last)
  const __nv_bfloat16* W1;               // [4h, h]
  const __nv_bfloat16* W2;               // [h, 4h]
};

struct SelectArgs {
  const float* Z;  int ldz;     // decoder tokens y = W_in m
  const float* KT; int ldkt;    // folded pointer keys
  const float* QS; int ldqs;    // folded self-attention queries (1/sqrt h inside)
  const float* KS; int ldks;    // self-attention keys
  const float* VT; int ldvt;    // folded values Wo_s Wv_s x
  const float* ln2_g; const float* ln2_b;
  float ln_eps;
  int stop_row, start_row;
  const float* stop_bias;
  int h, k_max, g;
  int* order; int* ep_count; float* margin; float* gap; int* rounds;
  int* err;
  // training-time pathway (Sec. 3.3): set score to also accumulate Eqs. 5-7
  // along the rollout (g = 1, keys in shared memory); NULL otherwise
  float* score;    // [sum N_b] s_i of Eq. 6, image-major rows
  float* kbar;     // [n_episodes] Eq. 7
  float inv_tau;   // 1 / pointer temperature
  float beta;      // discount of Eq. 6
  // pointer decoders of n_dec > 1 layers (g = 1)
  int n_dec;
  const DecLayerDev* dec;   // [n_dec] device array
  const float* KC;          // layer l's folded cross-attention keys at KC + 2 l h, values at + h (row stride ldz)
  float* dcache;            // self-attention rows (k | Wo Wv x) of layers 1..n_dec-1 per episode and position
  size_t dcache_ep;         // floats per episode: (n_dec - 1) (k_max + 1) 2h
};

int select_cluster_size(const BatchDesc& bd, int h, int k_max, bool* keys_in_smem, size_t* smem_bytes,
                        bool multi = false);
cudaError_t select_launch(const BatchDesc& bd, int n_episodes, const SelectArgs& a,
                          int cluster, bool keys_in_smem, size_t smem_bytes, cudaStream_t st);
// 3-D mRoPE (mrope.cu)
cudaError_t mrope_positions_launch(const BatchDesc& bd, const GridDesc& gd, const int* idx, int k_cap,
                                   const int* count, int* pos3, int T_cap, int* err, cudaStream_t st);
cudaError_t mrope_rows_launch(const float2* rope, int max_pos, int half, const int* pos3, int s1, int s2,
                              const int* T_dev, int T_cap, float2* rows, int* ident, int* err, cudaStream_t st);
// training-time pathway (train.cu)
cudaError_t soft_topk_launch(const BatchDesc& bd, int n_episodes, const float* score, const float* kbar, float tau,
                             float* alpha, float* k_out, cudaStream_t st);
cudaError_t vp_gate_launch(const void* X, const void* noise, const float* alpha, void* out, int rows, int D,
                           cudaStream_t st);
cudaError_t restore_launch(const BatchDesc& bd, const int* order, const int* ep_count, int k_max,
                           int* idx, int k_cap, int* count, int* err, cudaStream_t st);

// ------------------------------------------------------------- entry-point helpers (api.cu)
// Records a thread-local error message (sp_last_error) and returns `s`.
sp_status report(sp_status s, const char* fmt, ...);
// sp_select on an explicit scratch region (used by sp_select_noalloc).
sp_status select_with_workspace(const sp_selector* s, const sp_select_in* in, const sp_select_out* out,
                                void* ws, size_t ws_bytes, cudaStream_t st);

// ------------------------------------------------------------- compaction
cudaError_t compact_launch(const BatchDesc& bd, const void* X, int W_vis, const void* text, int W_txt,
                           const int* idx, int k_cap, const int* count, void* packed, int* cu,
                           int* pos, void* vis_packed, int* vis_row_map, int* vis_cu, int* vis_src, int T_cap,
                           int* err, cudaStream_t st);

}  // namespace sp
