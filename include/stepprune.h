/*
 * stepprune.h -- C ABI of the GB300 (sm_103a) StepPrune inference path.
 *
 * StepPrune (arXiv 2609.13804) prunes the visual prefix of a multimodal LLM by
 * sequential selection: a pointer decoder picks visual tokens one round at a
 * time, conditioned on what it already picked and on the text, until a learned
 * STOP action wins (Sec. 3.1-3.2, Eq. 2 and Eq. 4; grouped rounds of g tokens,
 * Sec. 3.5, Eq. 11).  The kept tokens are restored to native order and
 * physically gathered before the language-model prefill (Algorithm 1 steps 4-5).
 * This library runs that path on one GPU:
 *
 *   sp_select    text projection + cross-modal encoder (Eq. 3), candidate
 *                precompute, the sequential selection loop, restore.
 *   sp_compact   gather of the kept visual rows and the text rows into a packed
 *                variable-length buffer with cu_seqlens and positions.
 *   sp_project   the frozen multimodal projector on the kept rows, scattered
 *                into their packed slots.
 *   sp_prefill   the LM prefill over the packed prefix (hidden states after the
 *                final RMSNorm).
 *   sp_pipeline  all four, back to back on one stream.
 *
 * Conventions (all entry points):
 *   - Pointers marked DEVICE are device memory owned by the caller; HOST marks
 *     host memory read during the call only.  Matrices are row-major; weights
 *     use the nn.Linear layout [out_features, in_features].  bf16 data is
 *     passed as raw 16-bit patterns (void*).
 *   - Calls are asynchronous on the given stream and never synchronise the
 *     host.  Hot calls (sp_select, sp_compact, sp_project, sp_prefill,
 *     sp_pipeline) allocate nothing: scratch comes from the caller's workspace,
 *     sized by the matching *_workspace() query.  Handles allocate at create
 *     time only and free at destroy.
 *   - Sizes that depend on the selection (the kept counts, the packed length T)
 *     stay on the device; grids are sized from host-known caps and kernels
 *     skip rows past the device count, so no call reads results back.
 *   - A status is returned for every call; argument problems are detected on
 *     the host before any launch (nothing is launched then).  The message of
 *     the last failure on the calling thread is in sp_last_error().
 *   - Device-side failures (a bounded wait that ran out, an index out of
 *     range) set bits in the optional DEVICE int error word passed in the
 *     call; read it after synchronising (see SP_DEVERR_*).  Kernels never trap.
 *   - No C++ exception crosses the ABI.
 */
#ifndef STEPPRUNE_H
#define STEPPRUNE_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SP_API __attribute__((visibility("default")))
#else
#define SP_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

#define SP_ABI_VERSION 1

/* Limits checked on the host (SP_ERR_SHAPE when exceeded). */
#define SP_MAX_BATCH 256          /* images per call */
#define SP_MAX_ENC_LAYERS 4       /* cross-modal encoder blocks */
#define SP_MAX_DEC_LAYERS 4       /* pointer-decoder layers */
#define SP_MAX_LM_LAYERS 96       /* decoder layers of the LM */
#define SP_MAX_KMAX 1024          /* per-episode cap on retained tokens */
#define SP_MAX_NVIS 16384         /* visual tokens of one image */

typedef enum {
  SP_OK = 0,
  SP_ERR_INVALID_ARG = 1,   /* NULL where a pointer is required, bad enum, ... */
  SP_ERR_SHAPE = 2,         /* a size outside the supported set or a limit */
  SP_ERR_ALIGN = 3,         /* a device pointer not 16-byte aligned */
  SP_ERR_WORKSPACE = 4,     /* workspace NULL or smaller than *_workspace() */
  SP_ERR_CUDA = 5,          /* a CUDA runtime call failed (message has the code) */
  SP_ERR_TIMEOUT = 6,       /* reported by sp_device_error_status() */
  SP_ERR_UNSUPPORTED = 7,   /* device is not sm_103 / feature not built */
  SP_ERR_DEVICE = 8         /* reported by sp_device_error_status() */
} sp_status;

/* Bits of the DEVICE error word. */
#define SP_DEVERR_TIMEOUT 0x1   /* a bounded wait (mbarrier / flag) ran out */
#define SP_DEVERR_INDEX 0x2     /* an index outside its range was skipped */

typedef struct CUstream_st* sp_stream; /* a cudaStream_t; NULL is the legacy default stream */

/* Thread-local message of the last failed call ("" if none). */
SP_API const char* sp_last_error(void);
/* SP_ABI_VERSION of the loaded library. */
SP_API int sp_abi_version(void);
/* Maps a device error word read back by the caller to SP_OK / SP_ERR_TIMEOUT / SP_ERR_DEVICE. */
SP_API sp_status sp_device_error_status(int device_error_word);

/* ------------------------------------------------------------------------ */
/* Selector (Sec. 3.2: cross-modal encoder, STOP row, pointer decoder).      */
/* ------------------------------------------------------------------------ */

typedef struct {
  int D;             /* visual feature width = width of the candidate memory M; multiple of 128 */
  int D_text;        /* width of the prompt embeddings E_text */
  int h;             /* pointer-decoder width; multiple of 128 in 128..1024 */
  int n_enc_layers;  /* encoder blocks (the paper uses 2); 0..SP_MAX_ENC_LAYERS */
  int enc_head_dim;  /* encoder head dim: 64 or 128; D must be a multiple */
  int enc_ffn;       /* encoder MLP width (4 D in a ViT block) */
  float ln_eps;      /* LayerNorm epsilon */
  float g_text;      /* text gate g_text of E~ = g_text LN(W_p E) (1 at inference) */
  int n_dec_layers;  /* pointer-decoder layers, 1..SP_MAX_DEC_LAYERS (0 is read as 1) */
} sp_selector_cfg;

/*
 * Weights of the selector.  The encoder and text projection are bf16 (tensor
 * cores); the pointer decoder is fp32.  LayerNorm gain/bias pointers may be
 * NULL (gain 1 / bias 0).  All DEVICE; borrowed by the handle, so they must
 * outlive it (the handle keeps folded copies of the decoder matrices).
 *
 * Reading of the decoder (Sec. 3.2, Eq. 4; the paper fixes no layer count or
 * width): one pre-LN decoder layer of width h with single-head attention.  A
 * decoder token is y = W_in q with q_1 = s_start and q_{t+1} = M[a_t]; causal
 * self-attention gives u_t = y_t + Wo_s sum_i softmax_i(<Wq_s x_t, Wk_s x_i>/sqrt h)
 * Wv_s x_i with x_i = LN1(y_i); the pointer logits are the cross-attention
 * scores l_t(j) = <Wq_p LN2(u_t), Wk_p M_j>/sqrt h over the N+1 rows of
 * M = [H; s_stop], plus a per-episode stop_bias on the STOP row.
 *
 * With n_dec_layers = L > 1 the fields below (ln1, Wq_s .. Wo_s, ln2, Wq_p,
 * Wk_p) describe the LAST layer, and dec_lower[0 .. L-2] the layers before it,
 * each a whole pre-LN decoder layer of width h (Sec. 3.2: self-attention,
 * cross-attention to the memory, feed-forward network):
 *   a  = x + Wo_s SelfAttn(LN1(x))            causal over the history
 *   c  = a + Wo_c CrossAttn(LN2(a), M)        all N+1 rows of M, unmasked
 *   x' = c + W2 GELU(W1 LN3(c))               hidden width 4h, exact-erf GELU
 * x of layer 0 is y = W_in q; x' of layer L-2 enters the last layer.
 */
typedef struct {
  const float* ln1_g; const float* ln1_b;  /* [h] */
  const float* Wq_s; const float* Wk_s; const float* Wv_s; const float* Wo_s;  /* [h, h] fp32 */
  const float* ln2_g; const float* ln2_b;  /* [h] */
  const float* Wq_c; const float* Wo_c;    /* [h, h] fp32 */
  const float* Wk_c; const float* Wv_c;    /* [h, D] fp32 */
  const float* ln3_g; const float* ln3_b;  /* [h] */
  const void* W1;                          /* [4h, h] bf16 */
  const void* W2;                          /* [h, 4h] bf16 */
} sp_dec_layer_weights;

typedef struct {
  const void* W_p;                         /* [D, D_text] bf16 text projection */
  const float* ln_text_g; const float* ln_text_b;    /* [D] */
  const void* enc_wqkv[SP_MAX_ENC_LAYERS]; /* [3D, D] bf16, rows q|k|v */
  const void* enc_wo[SP_MAX_ENC_LAYERS];   /* [D, D] bf16 */
  const void* enc_w1[SP_MAX_ENC_LAYERS];   /* [enc_ffn, D] bf16 */
  const void* enc_w2[SP_MAX_ENC_LAYERS];   /* [D, enc_ffn] bf16 */
  const float* enc_ln1_g[SP_MAX_ENC_LAYERS]; const float* enc_ln1_b[SP_MAX_ENC_LAYERS];
  const float* enc_ln2_g[SP_MAX_ENC_LAYERS]; const float* enc_ln2_b[SP_MAX_ENC_LAYERS];
  const float* s_stop;                     /* [D] learned STOP embedding */
  const float* s_start;                    /* [D] learned START embedding (q_1) */
  const float* W_in;                       /* [h, D] decoder input projection */
  const float* ln1_g; const float* ln1_b;  /* [h] */
  const float* Wq_s; const float* Wk_s; const float* Wv_s; const float* Wo_s; /* [h, h] */
  const float* ln2_g; const float* ln2_b;  /* [h] */
  const float* Wq_p;                       /* [h, h] pointer query */
  const float* Wk_p;                       /* [h, D] pointer key */
  const sp_dec_layer_weights* dec_lower;   /* HOST [n_dec_layers - 1] (copied at creation; the
                                              DEVICE pointers inside are borrowed), or NULL */
} sp_selector_weights;

typedef struct sp_selector_s sp_selector;

/* Validates cfg, allocates the folded decoder matrices and encodes the weight
 * tensor maps.  Synchronous (uses the legacy stream once). */
SP_API sp_status sp_selector_create(const sp_selector_cfg* cfg, const sp_selector_weights* w,
                             sp_selector** out);
SP_API void sp_selector_destroy(sp_selector* s);

/*
 * One batch of images for selection.  Image b owns visual rows
 * [sum_{c<b} n_vis[c], +n_vis[b]) of X (or H) and text rows likewise of E_text.
 * Candidate groups: with group_size > 0 the candidates of an image are cut into
 * consecutive groups of group_size (the last may be shorter); each group is an
 * independent episode with its own mask, history, cap k_max and stop_bias, all
 * sharing s_start / s_stop; group_size 0 = one episode per image.  Episodes are
 * numbered image-major, group-minor.
 */
typedef struct {
  int B;                 /* images, 1..SP_MAX_BATCH */
  const int* n_vis;      /* HOST [B] visual tokens per image (N_b, 1..SP_MAX_NVIS) */
  const int* n_txt;      /* HOST [B] text tokens per image (L_b, >= 0) */
  const void* X;         /* DEVICE [sum N_b, D] bf16 visual tokens; ignored when H is set */
  const void* E_text;    /* DEVICE [sum L_b, D_text] bf16 prompt embeddings; ignored when H is set */
  const float* H;        /* DEVICE [sum N_b, D] fp32 encoded candidates, or NULL to run the
                            text projection and encoder on X / E_text (Eq. 3) */
  const float* stop_bias;/* DEVICE [n_episodes] fp32 added to the STOP logit */
  int group_size;        /* candidates per episode (0: whole image) */
  int g;                 /* visual tokens kept per non-STOP round (1..16); Eq. 11 */
  int k_max;             /* per-episode cap, 1..SP_MAX_KMAX */
} sp_select_in;

/*
 * Outputs.  idx row b holds image b's kept visual indices (image-local) in
 * ascending (native) order, then -1 up to k_cap.  k_cap must be at least the
 * largest possible count of an image: sum over its episodes of min(k_max, size).
 * order / ep_count / margin / gap are optional per-episode traces:
 *   order[e*k_max + i]   episode-local index taken i-th (step order)
 *   ep_count[e]          tokens kept by episode e
 *   margin[e*(k_max+1)+r] round r's smallest gap between consecutive values
 *                        among the top g+1 available visual logits and STOP
 *   gap[e*(k_max+1)+r]   round r's best available visual logit minus the raw
 *                        STOP logit (before stop_bias): STOP wins iff
 *                        stop_bias > gap, which calibrates stop_bias
 *   rounds[e]            evaluated rounds of episode e
 * Unwritten trace entries are left as they were.
 */
typedef struct {
  int* idx;          /* DEVICE [B, k_cap] */
  int k_cap;
  int* count;        /* DEVICE [B] kept tokens per image (K_b) */
  int* order;        /* DEVICE [n_episodes, k_max] or NULL */
  int* ep_count;     /* DEVICE [n_episodes] or NULL */
  float* margin;     /* DEVICE [n_episodes, k_max + 1] or NULL */
  float* gap;        /* DEVICE [n_episodes, k_max + 1] or NULL */
  int* rounds;       /* DEVICE [n_episodes] or NULL */
  float* memory;     /* DEVICE [sum N_b, D] fp32 or NULL: receives the candidate memory H
                        (the encoder output of Eq. 3, or a copy of the given H) */
  int* err;          /* DEVICE error word (SP_DEVERR_*) or NULL */
} sp_select_out;

/* Number of episodes of a batch (host arithmetic; -1 on bad arguments). */
SP_API int sp_num_episodes(int B, const int* n_vis, int group_size);
/* Workspace bytes sp_select needs for this batch (0 on bad arguments). */
SP_API size_t sp_select_workspace(const sp_selector* s, const sp_select_in* in);
/* Algorithm 1 steps 1-4 for every image of the batch (see sp_select_in).
 * A selector with n_dec_layers > 1 takes g = 1 only (each new history position
 * runs through every layer before the next decision; SP_ERR_UNSUPPORTED
 * otherwise, before any launch). */
SP_API sp_status sp_select(const sp_selector* s, const sp_select_in* in, const sp_select_out* out,
                    void* workspace, size_t workspace_bytes, sp_stream stream);

/*
 * sp_select without a caller workspace.  The paper has no counterpart: this is
 * for callers that cannot allocate device memory (a plug-in whose host
 * application owns all device memory, a plain-C caller with no allocator, a
 * path that may not pay for cudaMalloc).  It runs the same selection as
 * sp_select; its scratch is one static device array of
 * SP_SELECT_NOALLOC_SCRATCH_BYTES that every GPU loading the library holds
 * until exit.  Inputs and outputs are still the caller's.
 *   - A batch whose sp_select_workspace() exceeds that size is rejected with
 *     SP_ERR_WORKSPACE before any launch.
 *   - It calls no cudaMalloc / cudaFree and no allocating library routine.
 *   - The first call on a device looks up the array's device address (with
 *     that device current); make that first call before any stream capture.
 *   - All calls share the array and it keeps the last call's contents: calls
 *     whose GPU work overlaps (several streams or threads) race; serialise them.
 *   - The device address found by the first call is kept for the process's
 *     life: do not use this entry point across a device reset
 *     (cudaDeviceReset tears down the context the address belongs to).
 */
#define SP_SELECT_NOALLOC_SCRATCH_BYTES (64u << 20)
SP_API sp_status sp_select_noalloc(const sp_selector* s, const sp_select_in* in, const sp_select_out* out,
                                   sp_stream stream);

/* ------------------------------------------------------------------------ */
/* Training-time continuous pathway, forward only (Sec. 3.3, Eqs. 5-9).      */
/* ------------------------------------------------------------------------ */

/*
 * The trajectory aggregates of Eqs. 5-7, accumulated along the hard rollout:
 * at every evaluated step t of an episode, p_t = softmax(l_t / tau) over its
 * available candidates and STOP (l_t as in sp_select, stop_bias included:
 * pass zeros for the paper's training), and
 *   A_1 = 1,  A_{t+1} = A_t (1 - p_t(STOP))                       (Eq. 5)
 *   s_i  += A_t p_t(i) beta^t                                      (Eq. 6)
 *   Kbar += A_t (1 - p_t(STOP))                                    (Eq. 7)
 * The rollout is sp_select's (Eq. 4, hard argmax): it ends at the first hard
 * STOP, at k_max kept tokens or with only STOP left; later steps contribute
 * nothing.
 */
typedef struct {
  float tau;        /* pointer temperature, > 0 */
  float beta;       /* discount of Eq. 6, in (0, 1] */
  float* score;     /* DEVICE [sum N_b] fp32 out: s_i, same rows as X / H (4-byte aligned) */
  float* kbar;      /* DEVICE [n_episodes] fp32 out: Kbar per episode */
} sp_train_args;

/*
 * sp_select plus the aggregates above, in the same launches (same workspace
 * size as sp_select_workspace).  Requires g = 1 (one token per step, the
 * rollout the aggregates are defined on) and an episode size whose keys fit
 * the selection kernel's shared memory (up to 2,032 candidates per episode);
 * otherwise SP_ERR_UNSUPPORTED before any launch.  SP_ERR_INVALID_ARG for a
 * NULL score / kbar or tau <= 0 or beta outside (0, 1].
 */
SP_API sp_status sp_select_train(const sp_selector* s, const sp_select_in* in, const sp_select_out* out,
                                 const sp_train_args* train, void* workspace, size_t workspace_bytes,
                                 sp_stream stream);

/*
 * Eq. 8: alpha = SoftTopK_{k,tau}(s) per image, k = the batch mean of the
 * images' soft counts (an image's count is the sum of its episodes' Kbar),
 * detached, clamped to [0, N_b].  SoftTopK is the entropic optimal transport
 * of an image's scores (mass 1/N_b each) onto the anchors 0 and 1 with masses
 * (N_b - k, k) / N_b, cost (s_i - y)^2, regularisation tau; alpha_i is N_b
 * times token i's mass sent to anchor 1, which equals
 * sigmoid(2 (s_i - theta) / tau) with sum_i alpha_i = k (theta is solved for).
 *   n_vis / group_size: HOST, as in sp_select_in (episodes image-major)
 *   score: DEVICE [sum N_b] fp32, kbar: DEVICE [n_episodes] fp32
 *   alpha: DEVICE [sum N_b] fp32 out;  k_out: DEVICE [1] fp32 out or NULL
 * Errors: SP_ERR_INVALID_ARG / SP_ERR_SHAPE on bad sizes or pointers.
 */
SP_API sp_status sp_soft_topk(int B, const int* n_vis, int group_size, const float* score, const float* kbar,
                              float tau, float* alpha, float* k_out, sp_stream stream);

/*
 * Eq. 9: x~ = sqrt(alpha_r) x + sqrt(1 - alpha_r) eps for every row r, fp32
 * arithmetic, bf16 in and out.  X, noise, out: DEVICE [rows, D] bf16, 16-byte
 * aligned, D a multiple of 8; alpha: DEVICE [rows] fp32 (clamped to [0, 1]).
 * The Gaussian draws eps are the caller's.  out may alias X.
 */
SP_API sp_status sp_vp_gate(int rows, int D, const void* X, const void* noise, const float* alpha, void* out,
                            sp_stream stream);

/* ------------------------------------------------------------------------ */
/* Compaction (Algorithm 1 step 5: X_S = Gather(X, S), then [X_S; text]).    */
/* ------------------------------------------------------------------------ */

/*
 * Sequence b of the packed output is image b's kept visual rows (native order)
 * followed by its text rows; positions restart at 0 for every sequence.
 * T = cu_seqlens[B] is written on the device; T_cap = sum_b (min(n_vis[b], k_cap)
 * + n_txt[b]) bounds it.
 *   direct (vis_packed == NULL): W_vis must equal W_txt and visual rows go
 *     straight into their packed slots (no projector, or one already applied).
 *   projector mode (vis_packed != NULL): visual rows go to vis_packed, image-
 *     major and contiguous (vis_cu[b] is image b's first row), and
 *     vis_row_map[i] is the packed row that projected row i belongs to; the
 *     visual slots of packed are left for sp_project.
 */
typedef struct {
  int B;
  const int* n_vis;      /* HOST [B] */
  const int* n_txt;      /* HOST [B] */
  const void* X;         /* DEVICE [sum N_b, W_vis] bf16 */
  int W_vis;             /* multiple of 8 */
  const void* text;      /* DEVICE [sum L_b, W_txt] bf16 (LM-width prompt embeddings) */
  int W_txt;             /* multiple of 8 */
  const int* idx;        /* DEVICE [B, k_cap] from sp_select */
  int k_cap;
  const int* count;      /* DEVICE [B] */
} sp_compact_in;

typedef struct {
  void* packed;          /* DEVICE [T_cap, W_txt] bf16 */
  int* cu_seqlens;       /* DEVICE [B + 1] */
  int* pos;              /* DEVICE [T_cap] */
  void* vis_packed;      /* DEVICE [sum_b min(n_vis[b], k_cap), W_vis] bf16, or NULL (direct / index mode) */
  int* vis_row_map;      /* DEVICE [same rows] (projector and index modes) */
  int* vis_cu;           /* DEVICE [B + 1] (projector and index modes) */
  int* err;              /* DEVICE error word or NULL */
  int* vis_src;          /* DEVICE [same rows] int32, or NULL.  Index mode (vis_src set,
                            vis_packed NULL): no visual row is copied; vis_src[i] is the row of
                            X that kept visual row i comes from, and sp_project (io.vis_src)
                            gathers those rows itself: Alg. 1 step 5's gather folded into the
                            projector's operand load.  An invalid index gives vis_src -1. */
} sp_compact_out;

/* T_cap of a batch (host arithmetic; -1 on bad arguments). */
SP_API int sp_packed_cap(int B, const int* n_vis, const int* n_txt, int k_cap);
SP_API sp_status sp_compact(const sp_compact_in* in, const sp_compact_out* out, sp_stream stream);

/* ------------------------------------------------------------------------ */
/* Language model: projector + decoder-only prefill.                          */
/* ------------------------------------------------------------------------ */

typedef enum { SP_PROJ_NONE = 0, SP_PROJ_LINEAR = 1, SP_PROJ_MLP2_GELU = 2 } sp_proj_kind;

typedef struct {
  int n_layers;      /* 1..SP_MAX_LM_LAYERS */
  int d;             /* model width; multiple of 128 */
  int n_heads;       /* query heads */
  int n_kv_heads;    /* key/value heads; divides n_heads (GQA when smaller) */
  int head_dim;      /* 64 or 128 */
  int ffn;           /* SwiGLU width; multiple of 128 */
  int max_pos;       /* positions covered by the rotary table (> longest sequence) */
  float rope_theta;
  float rms_eps;
  int proj_kind;     /* sp_proj_kind */
  int proj_in;       /* visual width entering the projector */
  int proj_hidden;   /* hidden width of SP_PROJ_MLP2_GELU */
  int mrope_section[3]; /* 3-D mRoPE (the Qwen2.5-VL backbone, Sec. 1): rotation pairs given to the
                           (t, h, w) position components, consecutive from pair 0; the three sum
                           to head_dim / 2, each even.  All zero: 1-D RoPE on pos. */
} sp_model_cfg;

/*
 * Weights (DEVICE, borrowed; bf16 unless stated).  Per layer:
 *   wqkv  [(n_heads + 2 n_kv_heads) head_dim, d]  rows q | k | v
 *   wo    [d, n_heads head_dim]
 *   wgu   [2 ffn, d]  rows gate | up   (SwiGLU: down(silu(gate x) * up x))
 *   wdown [d, ffn]
 *   attn_norm / mlp_norm  fp32 [d] RMSNorm gains, or NULL (1)
 * final_norm fp32 [d] or NULL.  Projector: proj_w1 [proj_hidden or d, proj_in],
 * proj_w2 [d, proj_hidden] (SP_PROJ_MLP2_GELU only).
 */
typedef struct {
  const void* wqkv[SP_MAX_LM_LAYERS];
  const void* wo[SP_MAX_LM_LAYERS];
  const void* wgu[SP_MAX_LM_LAYERS];
  const void* wdown[SP_MAX_LM_LAYERS];
  const float* attn_norm[SP_MAX_LM_LAYERS];
  const float* mlp_norm[SP_MAX_LM_LAYERS];
  const float* final_norm;
  const void* proj_w1;
  const void* proj_w2;
} sp_model_weights;

typedef struct sp_model_s sp_model;

/* Validates cfg, uploads the rotary table (fp64 on the host, stored fp32) and
 * encodes the weight tensor maps.  Synchronous. */
SP_API sp_status sp_model_create(const sp_model_cfg* cfg, const sp_model_weights* w, sp_model** out);
SP_API void sp_model_destroy(sp_model* m);

/*
 * Projector on the kept rows (Sec. 3.3, last paragraph: restored, then
 * projected): packed[vis_row_map[i]] = P(x_i) for i < vis_cu[B] (device
 * count), P = W1 x, or W2 GELU(W1 x), with x_i = vis_packed[i], or, when
 * vis_src is given, x_i = X[vis_src[i]] read by the first GEMM's operand loads
 * (row-gather TMA) so that the kept rows are never copied.  rows_cap bounds
 * vis_cu[B].
 */
typedef struct {
  int B;
  int rows_cap;
  const void* vis_packed;   /* DEVICE [rows_cap, proj_in] bf16 (ignored with vis_src) */
  const int* vis_row_map;   /* DEVICE [rows_cap] */
  const int* vis_cu;        /* DEVICE [B + 1] */
  void* packed;             /* DEVICE [T_cap, d] bf16 (visual slots written) */
  int* err;
  const void* X;            /* DEVICE [rows_X, proj_in] bf16 visual tokens (with vis_src) */
  int rows_X;               /* rows of X (with vis_src) */
  const int* vis_src;       /* DEVICE [rows_cap] rows of X (sp_compact's index mode), or NULL */
} sp_project_io;

SP_API size_t sp_project_workspace(const sp_model* m, int rows_cap);
SP_API sp_status sp_project(const sp_model* m, const sp_project_io* io, void* workspace,
                     size_t workspace_bytes, sp_stream stream);

/*
 * Prefill of the packed sequences: the frozen LM run over the pruned prefix
 * that Algorithm 1 hands it (Sec. 3.3, last paragraph: the kept tokens,
 * restored to native order and projected, precede the text; Sec. 1: the
 * prefill cost the selection removes is that of the dropped visual tokens).
 * The layers are those of the evaluated backbones (Sec. 4.1): causal attention
 * within each sequence (cu_seqlens), grouped-query heads, rotary positions
 * pos, pre-RMSNorm Llama-style layers with SwiGLU, and the final RMSNorm.
 * hidden rows t < T = cu_seqlens[B] are written; rows >= T are untouched.  residual (optional) receives the last residual stream (fp32,
 * before the final norm).  kv (optional) receives the key / value cache the
 * generation that follows reads (sp_decode): per layer l, sequence b and
 * position p = pos[row] the rotated key at
 *   kv + (((l * 2 + 0) * B + b) * kv_S_cap + p) * (n_kv_heads * head_dim)
 * and the value at the same offset with 1 in place of 0 (bf16).  Positions
 * must be < kv_S_cap (else SP_DEVERR_INDEX).
 * With an mRoPE model (mrope_section set), pos3 gives every row's rotary
 * (t, h, w) position (sp_mrope_positions writes it for a pruned batch); pos is
 * then only the row's index within its sequence (its cache slot).  A rotary
 * position >= max_pos sets SP_DEVERR_INDEX.
 */
typedef struct {
  int B;
  int T_cap;                /* bound on cu_seqlens[B] */
  int max_seqlen_cap;       /* bound on every sequence length */
  const void* x;            /* DEVICE [T_cap, d] bf16 packed LM input */
  const int* cu_seqlens;    /* DEVICE [B + 1] */
  const int* pos;           /* DEVICE [T_cap] */
  float* hidden;            /* DEVICE [T_cap, d] fp32 output */
  float* residual;          /* DEVICE [T_cap, d] fp32 or NULL */
  int* err;
  void* kv;                 /* DEVICE [n_layers][2][B][kv_S_cap][n_kv_heads * head_dim] bf16, or NULL */
  int kv_S_cap;             /* positions per sequence in kv */
  const int* pos3;          /* DEVICE [T_cap, 4] int32 (t, h, w, unused); required iff mRoPE, else NULL */
} sp_prefill_io;

/*
 * mRoPE positions of a pruned batch (reading of Sec. 3.3's last paragraph: the
 * kept tokens are restored to native order so that the backbone's positional
 * convention holds).  Image b's N_b tokens form a grid of ceil(N_b / grid_w[b])
 * rows of grid_w[b] tokens at time 0; a kept token idx keeps its grid position
 * (0, idx / grid_w, idx % grid_w); the text after it continues on all three
 * components from max(rows, grid_w[b]) (the unpruned image block's largest
 * position + 1).  Row cu + j of sequence b (cu = sum over earlier images of
 * count + n_txt, the packing of sp_compact) gets the j-th position.
 *   n_vis, n_txt, grid_w: HOST [B];  idx [B, k_cap], count [B]: DEVICE (sp_select)
 *   pos3: DEVICE [T_cap, 4] int32 out (rows >= the packed length untouched)
 * Errors: bad sizes -> SP_ERR_SHAPE; on the device, an index outside its image
 * or a row >= T_cap sets SP_DEVERR_INDEX (the row is skipped).
 */
SP_API sp_status sp_mrope_positions(int B, const int* n_vis, const int* n_txt, const int* grid_w, const int* idx,
                                    int k_cap, const int* count, int* pos3, int T_cap, int* err, sp_stream stream);

SP_API size_t sp_prefill_workspace(const sp_model* m, int T_cap, int max_seqlen_cap);
SP_API sp_status sp_prefill(const sp_model* m, const sp_prefill_io* io, void* workspace,
                     size_t workspace_bytes, sp_stream stream);

/*
 * One generation step after the prefill (the decode whose per-token latency
 * the pruned prefix lowers): every sequence b appends one token x[b] at
 * position lens[b], which attends to the cached keys / values 0..lens[b]-1
 * (written by sp_prefill's kv, or by earlier steps) and to itself; the layers
 * are the prefill's, applied to that one row.  The step writes the new
 * token's rotated key / value into the cache at position lens[b], the final
 * RMSNorm of its last residual into hidden[b], and then increments lens[b]
 * (on the device, so steps chain without a host round trip).
 * Errors: a position >= kv_S_cap sets SP_DEVERR_INDEX (nothing is written
 * for that sequence's cache row); more than 8 query heads per key / value
 * head -> SP_ERR_UNSUPPORTED.  max_len_cap sizes the attention's key split
 * only: a longer sequence is still attended in full (its ranges grow).
 */
typedef struct {
  int B;                    /* sequences, as in the prefill that wrote kv */
  const void* x;            /* DEVICE [B, d] bf16: the new token of each sequence */
  int* lens;                /* DEVICE [B] int32: cached positions per sequence; incremented */
  void* kv;                 /* DEVICE cache, layout of sp_prefill_io.kv */
  int kv_S_cap;             /* positions per sequence in kv */
  int max_len_cap;          /* bound on lens[b] + 1 (sizes the attention launch) */
  float* hidden;            /* DEVICE [B, d] fp32 output */
  int* err;
  int* rope_pos;            /* DEVICE [B] int32 rotary position of each new token, or NULL (= lens);
                               incremented with lens.  After an mRoPE prefix: the position the
                               next text token takes (on all three components, so the 1-D
                               rotation at that position) */
} sp_decode_io;

SP_API size_t sp_decode_workspace(const sp_model* m, int B);
SP_API sp_status sp_decode(const sp_model* m, const sp_decode_io* io, void* workspace, size_t workspace_bytes,
                           sp_stream stream);

/* ------------------------------------------------------------------------ */
/* The whole path: select -> compact -> project -> prefill.                  */
/* ------------------------------------------------------------------------ */

/*
 * Algorithm 1 (Sec. 3.5) end to end on the device, followed by the prefill
 * over its result: the text projection and the encoder (Eq. 3), the pointer
 * rounds of Eq. 4 / Eq. 11 with the STOP action per episode, the restore to
 * native order, the gather into packed sequences [kept visual rows; text
 * rows] (Sec. 3.3, last paragraph), the projector on the kept rows, and the
 * LM prefill of sp_prefill.  One stream, no host synchronisation: sizes that
 * depend on the selection stay on the device (grids are sized from caps).
 * Outputs: idx / count as sp_select's, cu_seqlens as sp_compact's, hidden as
 * sp_prefill's.  Errors: the union of those of the four calls; the
 * workspace must hold sp_pipeline_workspace() bytes (SP_ERR_WORKSPACE).
 */
typedef struct {
  sp_select_in sel;          /* X and E_text required (H ignored); E_text is also the
                                text rows of the LM input, so D_text must equal d */
  int k_cap;                 /* row stride of idx */
  int* idx;                  /* DEVICE [B, k_cap] */
  int* count;                /* DEVICE [B] */
  int* cu_seqlens;           /* DEVICE [B + 1] */
  float* hidden;             /* DEVICE [T_cap, d] fp32 (T_cap = sp_packed_cap(...)) */
  int* err;                  /* DEVICE error word or NULL */
} sp_pipeline_io;

SP_API size_t sp_pipeline_workspace(const sp_selector* s, const sp_model* m, const sp_pipeline_io* io);
SP_API sp_status sp_pipeline(const sp_selector* s, const sp_model* m, const sp_pipeline_io* io,
                      void* workspace, size_t workspace_bytes, sp_stream stream);

/*
 * The same path from HOST buffers: copies X, E_text and stop_bias (HOST, best
 * pinned) into the workspace, runs sp_pipeline, and copies idx, count,
 * cu_seqlens and the T_cap hidden rows back into the HOST outputs, all on
 * `stream`.  The host buffers must stay valid until the stream reaches the end
 * of the call.  The io's DEVICE pointer fields are ignored; host_* are used.
 */
typedef struct {
  sp_select_in sel;          /* X, E_text, stop_bias are HOST pointers here */
  int k_cap;
  int* host_idx;             /* HOST [B, k_cap] */
  int* host_count;           /* HOST [B] */
  int* host_cu_seqlens;      /* HOST [B + 1] */
  float* host_hidden;        /* HOST [T_cap, d] */
} sp_pipeline_host_io;

SP_API size_t sp_pipeline_host_workspace(const sp_selector* s, const sp_model* m,
                                  const sp_pipeline_host_io* io);
SP_API sp_status sp_pipeline_host(const sp_selector* s, const sp_model* m, const sp_pipeline_host_io* io,
                           void* workspace, size_t workspace_bytes, sp_stream stream);

/* ------------------------------------------------------------------------ */
/* Failure-detection self-test (the paper has no counterpart).               */
/* ------------------------------------------------------------------------ */

/*
 * Every wait in this library's kernels is bounded (2 s): one that runs out
 * sets SP_DEVERR_TIMEOUT in the call's error word and the kernel returns, so a
 * lost arrival never hangs the GPU.  This call runs the two wait helpers the
 * kernels use, with limit_us microseconds (1 .. 2,000,000) in place of 2 s:
 *   out[0] = 1 if a wait on an mbarrier completed, 0 if it timed out,
 *   out[1] = 1 if a wait for *flag == 1 completed, 0 if it timed out.
 * The mbarrier gets no arrival (so the wait runs out) unless `complete` is
 * non-zero; the flag wait completes iff the caller's DEVICE int *flag is 1.
 * A timeout ORs SP_DEVERR_TIMEOUT into *err (DEVICE, may be NULL);
 * sp_device_error_status() maps it to SP_ERR_TIMEOUT.  The stream and the
 * context stay usable.  flag, out: DEVICE.  Asynchronous on `stream`.
 * Errors: SP_ERR_INVALID_ARG (NULL flag / out), SP_ERR_SHAPE (limit out of
 * range), SP_ERR_CUDA.
 */
SP_API sp_status sp_wait_probe(const int* flag, unsigned int limit_us, int complete, int* out, int* err,
                               sp_stream stream);

/* ------------------------------------------------------------------------ */
/* Per-kernel timing (CUDA events recorded around every launch).             */
/* ------------------------------------------------------------------------ */

typedef enum {
  SP_K_GEMM = 0, SP_K_SGEMM = 1, SP_K_ATTN = 2, SP_K_NORM = 3, SP_K_SELECT = 4,
  SP_K_RESTORE = 5, SP_K_COMPACT = 6, SP_K_MISC = 7, SP_K_TRAIN = 8, SP_K_COUNT = 9
} sp_kernel_kind;

/* Starts (capacity > 0) or stops (0) recording launch events; host-allocated. */
SP_API sp_status sp_profile_begin(int capacity);
/* Synchronises on the recorded events and returns, per sp_kernel_kind, the
 * summed milliseconds, launch counts and algorithmic flops / bytes. */
SP_API sp_status sp_profile_end(double* ms, long long* launches, double* flops, double* bytes);

#ifdef __cplusplus
}
#endif
#endif /* STEPPRUNE_H */
