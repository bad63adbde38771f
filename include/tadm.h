/*
 * tadm.h - C ABI of the GB300 (sm_103a) implementation of TADM's
 * anchor-cache reverse-diffusion sampling loop (Time-Anchored Diffusion
 * Language Models).
 *
 * The method (paper §3): a denoising network is split into a shared network
 * S, an expensive anchor network A, a small fusion module Phi and a light
 * denoiser D.  The anchor latent h = A(S(z)) is refreshed once every K
 * reverse steps and cached in HBM; every step encodes the current canvas
 * c = S(z), fuses it with the stale cache, h~ = Phi(c, h_cache)
 * (Eq. stale-anchor-fusion), and denoises, x = D(h~) (Alg. 1).  The default
 * sampler unmasks the most confident masked positions of the active block;
 * the paper's own samplers, ReMDM remasking (App. C.2) and the entropy-bound
 * sampler with self-conditioning (App. C.1, Alg. 2), have entry points of
 * their own at the end of this header.
 *
 * Conventions for every call:
 *  - Pointers named "device" are CUDA device pointers; the caller owns and
 *    frees all of them (the library allocates no device memory).  "host"
 *    pointers are plain host memory.
 *  - Token ids are int32.  MASK is vocab - 1.  Every id the caller passes
 *    must lie in [0, vocab - 1].
 *  - Matrices are row-major.  A projection from n_in to n_out features is a
 *    weight [n_out, n_in] (y = x W^T).
 *  - Calls that take a stream only enqueue work on it and return at once;
 *    kernels that give up a bounded wait set a device status word that
 *    tadm_sync_status() turns into TADM_ERR_TIMEOUT.  Argument errors are
 *    detected on the host, before anything is enqueued.
 *  - No call throws, aborts or exits.  On error the returned status is
 *    non-zero and tadm_last_error() describes it.
 *  - A handle must not be used by two host threads at once.
 */
#ifndef TADM_H
#define TADM_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define TADM_API __attribute__((visibility("default")))
#else
#define TADM_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t; NULL means the legacy default stream. */
typedef struct CUstream_st* tadm_stream;

typedef enum {
  TADM_OK = 0,
  TADM_ERR_INVALID_ARG = 1, /* bad shape, size, pointer or alignment */
  TADM_ERR_UNSUPPORTED = 2, /* valid model, but a shape this build does not run */
  TADM_ERR_CUDA = 3,        /* a CUDA runtime call failed */
  TADM_ERR_OOM = 4,         /* the bound workspace is smaller than required */
  TADM_ERR_TIMEOUT = 5,     /* a kernel gave up a bounded wait */
  TADM_ERR_STATE = 6        /* call out of order (no workspace, context full, ...) */
} tadm_status;

/*
 * Model description (paper §3.1, App. C.1, App. C.2).
 *  glu:     0 = SwiGLU (SiLU gate), 1 = GeGLU (tanh-approximate GELU gate).
 *  n_shared, n_anchor, n_denoise: L_S, L_A, L_D of Eq. (anchor-cache-compute);
 *           S is the token embedding followed by n_shared layers.
 *  fusion:  0 = gated residual MLP (App. C.2):
 *              u = [LN(c); LN(h)], g = sigmoid(W_g u + b_g),
 *              Delta = W_2 GELU(W_1 u + b_1) + b_2, h~ = LN(h + g * Delta);
 *           1 = paired attention with cached shallow state (App. C.1,
 *              Eqs. paired-attention-difference, stale-anchor-fusion-app);
 *           2 = off: the denoiser reads the cached anchor output itself,
 *              h~ = h' (the naive stale-anchor reuse baseline of App. D,
 *              Table naive-vs-tadm-posttrain); no fusion weights.
 *  fusion_rank, fusion_heads: r and the mixer heads of fusion 1.
 *  dtype:   0 = fp32 weights and activations, 1 = bf16 weights and GEMM
 *           operands (fp32 accumulation, fp32 residual stream).
 *  tied_lm_head: 1 = the output head reuses the embedding matrix.
 *  Gemma-3 layer details of the Post-train backbone (App. C.1 names a
 *  Gemma-3 based model and gives no layer details; these follow the public
 *  Gemma-3 architecture; all zero = a plain pre-norm layer):
 *  sliding_window: W > 0: a query at position p of a local layer sees only
 *           keys at positions j with p - j < W (besides the causal rule of
 *           prefill / commit passes); 0 = local layers see every key.
 *  global_every: g > 0: layer i of the whole backbone (the L_S shared, then
 *           the L_A anchor, then the L_D denoiser layers, 0-based) is global
 *           iff (i + 1) % g == 0, otherwise local; g = 0: every layer global.
 *           Global layers see every key.
 *  qk_norm: 1 = RMSNorm over head_dim of every Q and K head (gains q_norm,
 *           k_norm of the layer), before RoPE.
 *  sandwich_norm: 1 = each sub-block's output is RMS-normalised (gains
 *           post_attn_norm, post_ffn_norm) before the residual add.
 *  rope_theta_global: RoPE base of global layers (0 = rope_theta); local
 *           layers use rope_theta.
 *  qkv_split: bf16 models only: 1 = the normalised input of every QKV
 *           projection enters the tensor cores as two bf16 terms, hi =
 *           bf16(n) and lo = bf16(n - hi), both multiplying the same weight
 *           tiles (the projection then costs twice the MMA work); its input
 *           is carried to about 16 significant bits instead of 8.  The
 *           attention logits are the most rounding-sensitive quantity of the
 *           backbone, and this keeps the committed tokens of a
 *           teacher-forced generation on those of the exact model.
 */
typedef struct {
  int32_t vocab, d_model, n_heads, n_kv_heads, head_dim, ffn;
  int32_t glu;
  int32_t n_shared, n_anchor, n_denoise;
  int32_t fusion;
  int32_t fusion_rank, fusion_heads;
  int32_t dtype;
  int32_t tied_lm_head;
  float norm_eps, rope_theta;
  int32_t sliding_window, global_every, qk_norm, sandwich_norm;
  float rope_theta_global;
  int32_t qkv_split;
} tadm_config;

typedef struct tadm_handle tadm_handle;

/* ---------------------------------------------------------------- weights --
 * The model's parameters are passed as an array of device pointers in the
 * order this inventory lists them.  Element type: fp32 when dtype = 0, bf16
 * when dtype = 1.  Each tensor is contiguous, row-major [rows, cols] (vectors
 * have cols = 1... rows = length) and 16-byte aligned.
 *
 * Inventory: "embed" [V, d]; then for net in (shared, anchor, denoise) and
 * each layer i: "<net>.<i>.attn_norm" [d], ".wqkv" [(Hq + 2 Hkv) hd, d]
 * (rows: Q heads, K heads, V heads), with qk_norm ".q_norm" [hd] and
 * ".k_norm" [hd], ".wo" [d, Hq hd], with sandwich_norm ".post_attn_norm"
 * [d], ".ffn_norm" [d], ".wgu" [2F, d] (rows: gate, then up), ".wdown"
 * [d, F], with sandwich_norm ".post_ffn_norm" [d]; then the fusion
 * parameters; "final_norm" [d]; "lm_head" [V, d] unless tied.
 */
/* Number of weight tensors of cfg, or -1 if cfg is invalid. */
TADM_API int tadm_weight_count(const tadm_config* cfg);
/* Name (NUL-terminated, truncated to name_cap) and shape of tensor `index`.
 * Vectors report cols = 1.  INVALID_ARG for a bad index or config. */
TADM_API tadm_status tadm_weight_info(const tadm_config* cfg, int index, char* name, int name_cap,
                             int64_t* rows, int64_t* cols);

/* ----------------------------------------------------------------- handle --
 * tadm_create validates cfg and copies the weight pointers (the weights must
 * stay valid for the handle's life).  Sizes fix the workspace:
 *   max_batch: sequences per call;
 *   max_rows:  canvas rows per sequence in one step (block_len in block mode,
 *              prompt + generation length in single-block mode);
 *   max_ctx:   block mode: positions per sequence that hold K/V (the prompt,
 *              every committed block and the active block, i.e. at least
 *              prompt + generation length); 0 when only the single-block
 *              mode is used.
 */
TADM_API tadm_status tadm_create(const tadm_config* cfg, const void* const* weights, int n_weights,
                        int max_batch, int max_rows, int max_ctx, tadm_handle** out);
TADM_API void tadm_destroy(tadm_handle* h);
TADM_API const char* tadm_last_error(const tadm_handle* h);
TADM_API const char* tadm_status_string(tadm_status s);

/* Device workspace: activations, KV caches, the internal anchor cache of
 * tadm_generate and the status word.  Caller allocates >= *bytes, 256-byte
 * aligned, and binds it before any compute call.  Binding synchronises the
 * device once (it fills the RoPE table) and drops the CUDA graph that
 * tadm_generate may hold, so nothing recorded on the previous workspace is
 * replayed; the previous workspace may be freed once the work queued on it
 * has finished. */
TADM_API tadm_status tadm_workspace_size(const tadm_handle* h, size_t* bytes);
TADM_API tadm_status tadm_bind_workspace(tadm_handle* h, void* dev_ptr, size_t bytes);

/* Bytes of one anchor cache for `batch` sequences of `rows` canvas rows
 * (fusion 0 and 2: h, fp32 [batch*rows, d]; fusion 1: H0, s_C, s_H, Z0, U and
 * phi(Z0, U)).  Caller-allocated, device, 256-byte aligned. */
TADM_API tadm_status tadm_cache_size(const tadm_handle* h, int batch, int rows, size_t* bytes);

/* ------------------------------------------------------ one step of Alg. 1 --
 * Block mode: tadm_reset, tadm_prefill(prompt), then per block the steps on
 * the block's canvas rows, then tadm_commit_block.  Single-block mode:
 * tadm_reset then steps on the whole canvas (context stays empty).
 * x_t: device int32 [batch, rows] canvas of the active rows, positions
 * ctx .. ctx + rows - 1 where ctx is the committed context length.
 */
TADM_API tadm_status tadm_reset(tadm_handle* h, int batch);

/* Causal fresh pass S -> A -> Phi(c, A(c)) -> D over the prompt; every
 * layer's K, V join the context (App. C.1, encoder prefill).
 * prompt: device int32 [batch, prompt_len]. */
TADM_API tadm_status tadm_prefill(tadm_handle* h, const int32_t* prompt, int batch, int prompt_len,
                         tadm_stream stream);

/* Refresh branch of Alg. 1: h_cache <- A(S(x_t)).  `t` is the step index i of
 * Alg. 1 (informational; time conditioning is off).  h_cache: device, at
 * least tadm_cache_size(batch, rows) bytes. */
TADM_API tadm_status tadm_anchor_forward(tadm_handle* h, const int32_t* x_t, int batch, int rows, int t,
                                void* h_cache, tadm_stream stream);

/* Optional outputs of a denoising step (device pointers, each may be NULL):
 *  logits:   fp32 [batch*rows, vocab] (written only if non-NULL; the fast
 *            path never materialises them);
 *  conf:     fp32 [batch*rows] max softmax probability over ids != MASK;
 *  tok:      int32 [batch*rows] its argmax (lowest id on ties);
 *  selected: int32 [batch, k_n] positions unmasked this step, ascending rank,
 *            -1 padded;
 *  fused:    fp32 [batch*rows, d] the fused latent h~ = Phi(c, h_cache) that
 *            enters D. */
typedef struct {
  float* logits;
  float* conf;
  int32_t* tok;
  int32_t* selected;
  float* fused;
} tadm_step_outputs;

/* One reverse step: c = S(x_t), h~ = Phi(c, h_cache), logits = head(D(h~)),
 * then the sampler unmasks k_n = floor((n+1) G / T) - floor(n G / T)
 * positions per sequence (n = T - t, G = n_masked_at_start): the masked
 * positions of largest confidence, ties toward the lower position.  Tokens
 * already unmasked are never changed (carry-over), MASK is never predicted
 * (zero-masking).  x_t is updated in place.  `out` may be NULL. */
TADM_API tadm_status tadm_denoise_step(tadm_handle* h, int32_t* x_t, int batch, int rows, int t, int T,
                              int n_masked_at_start, const void* h_cache,
                              const tadm_step_outputs* out, tadm_stream stream);

/* Causal fresh pass over a finalised block; its K, V join the context. */
TADM_API tadm_status tadm_commit_block(tadm_handle* h, const int32_t* x_block, int batch, int rows,
                              tadm_stream stream);

/* Whole generation (Alg. 1 per block).  prompt: device int32 [batch,
 * prompt_len]; out: device int32 [batch, prompt_len + gen_len], the final
 * canvas.  block_len = 0: one block over the whole canvas (bidirectional,
 * no KV context); else gen_len % block_len == 0 and the prompt is prefilled.
 * The anchor refreshes at n = 0, K, 2K, ... of every block.  The second call
 * with the same sizes, prompt, out and workspace is captured into a CUDA
 * graph on an internal stream and later identical calls replay it (ordered
 * after the caller's stream by events); TADM_GRAPH=0 in the environment
 * keeps every call eager. */
TADM_API tadm_status tadm_generate(tadm_handle* h, const int32_t* prompt, int batch, int prompt_len,
                          int32_t* out, int gen_len, int steps_per_block, int K, int block_len,
                          tadm_stream stream);

/* Waits for the last stream used by h, then reports TADM_ERR_TIMEOUT if a
 * kernel gave up a bounded wait since the last reset of the status word
 * (tadm_generate and tadm_reset clear it), TADM_ERR_CUDA on a CUDA error. */
TADM_API tadm_status tadm_sync_status(tadm_handle* h);

/* ------------------------------------------------------------- accounting --
 * Layer evaluations and anchor calls issued by reverse steps since the last
 * tadm_reset / tadm_generate (prefill and commit passes are counted apart),
 * the quantities of Eq. (anchor-cache-compute). */
typedef struct {
  int64_t shared_layers, anchor_layers, denoise_layers;
  int64_t anchor_calls, denoise_steps;
  int64_t commit_passes;
  int64_t kernel_launches; /* CUDA kernels this handle launched */
} tadm_counters;
TADM_API tadm_status tadm_get_counters(const tadm_handle* h, tadm_counters* out);

/* Timing probe.  While enabled, every GEMM, attention and normalisation
 * launch of the handle is bracketed by two CUDA events recorded on its
 * stream (a pool of up to `max_launches` pairs, created here), and the
 * algorithmic work of GEMMs (2*M*N*K) and attention (4*rows*keys*hd per
 * head) is noted.  tadm_probe_read waits for the last event and returns the
 * number of bracketed GEMM launches, their summed duration (ms) and summed
 * FLOPs, then clears the records.  tadm_probe_enable(h, 0) frees the events. */
TADM_API tadm_status tadm_probe_enable(tadm_handle* h, int max_launches);
TADM_API tadm_status tadm_probe_read(tadm_handle* h, int64_t* launches, double* total_ms, double* total_flops);
/* The records split by kind: GEMM epilogues 0 plain, 1 residual, 2 QKV +
 * RoPE, 3 GLU, 4 fusion gate/hidden, 5 fusion output, 6 output head,
 * 7..10 paired-attention fusion; 11 attention; 12 RMSNorm / LayerNorm
 * launches; 13 attention over fewer than 128 canvas rows (block steps).
 * Arrays of n_kinds entries.  bytes (optional, may be NULL): the algorithmic
 * bytes of the GEMM records (A and B read once, the output written once, the
 * residual stream read and written by residual epilogues; for the output
 * head only A and B, its logits never reach memory).  Call before
 * tadm_probe_read, which clears the records. */
TADM_API tadm_status tadm_probe_breakdown(tadm_handle* h, int n_kinds, int64_t* launches, double* ms,
                                          double* flops, double* bytes);

/* Plan of tadm_generate (host only, no GPU): the ordered phases it issues.
 * kind: 0 prefill, 1 anchor refresh, 2 denoise step, 3 commit.  For kinds 1
 * and 2, n is the step within the block and k the positions unmasked
 * (kind 2).  Writes at most `cap` events; *n_events gets the full count. */
typedef struct {
  int32_t kind, block, n, k;
} tadm_plan_event;
TADM_API tadm_status tadm_plan(int prompt_len, int gen_len, int steps_per_block, int K, int block_len,
                      tadm_plan_event* events, int cap, int* n_events);

/* Eq. (anchor-cache-compute): C_full = T (L_S + L_A + L_D) and
 * C_cache = T (L_S + L_D) + ceil(T / K) L_A. */
TADM_API tadm_status tadm_layer_cost(int L_S, int L_A, int L_D, int T, int K, int64_t* c_full,
                            int64_t* c_cache);

/* --------------------------------------------------------- building blocks --
 * The kernels of the path, exposed for unit parity tests and benchmarks.
 * They use no handle and need no workspace; all pointers are device pointers.
 */
/* C[M, N] = A[M, K] B[N, K]^T.  dtype 1: A, B bf16 (tcgen05 tensor cores,
 * fp32 accumulate); dtype 0: fp32 (CUDA cores).  c_dtype: 0 fp32, 1 bf16.
 * Row strides lda, ldb, ldc in elements; rows 16-byte aligned. */
TADM_API tadm_status tadm_gemm(const void* A, const void* B, void* C, int M, int N, int K, int lda, int ldb,
                      int ldc, int dtype, int c_dtype, tadm_stream stream);

/* Per row of fp32 logits [rows, vocab]: tok = argmax over ids != mask_id
 * (lowest id on ties), conf = 1 / sum_v exp(l_v - l_tok). */
TADM_API tadm_status tadm_confidence(const float* logits, int rows, int vocab, int mask_id, float* conf,
                            int32_t* tok, tadm_stream stream);

/* Sampler update of z [batch, rows] (row stride ldz) from per-position conf
 * and tok ([batch, rows], dense): unmask the k masked positions of largest
 * conf in each sequence (ties -> lower position); selected [batch, k] or
 * NULL. */
TADM_API tadm_status tadm_topk_unmask(int32_t* z, int ldz, const float* conf, const int32_t* tok, int batch,
                             int rows, int k, int mask_id, int32_t* selected, tadm_stream stream);

/* Fused output head + confidence (the sampler's input, paper App. B.1.1
 * zero-masking): for each row of x [rows, d], logits = x W^T over W
 * [vocab, d] are reduced inside the GEMM epilogue to per-column-tile
 * (max, sum exp, argmax) partials, which a second kernel merges into
 * tok = argmax over ids != mask_id (lowest id on ties) and
 * conf = 1 / sum_v exp(l_v - l_tok).  The logits never reach memory.
 * dtype 1: x, W bf16 (tcgen05); 0: fp32.  scratch: device, at least
 * tadm_head_scratch_size() bytes, holds the partials; it needs no
 * initialisation and its contents are meaningless after the call. */
TADM_API tadm_status tadm_head_scratch_size(int rows, int vocab, int dtype, size_t* bytes);
TADM_API tadm_status tadm_head_confidence(const void* x, const void* w, int rows, int d, int vocab, int mask_id,
                                          int dtype, void* scratch, size_t scratch_bytes, float* conf,
                                          int32_t* tok, tadm_stream stream);

/* tadm_head_confidence without caller scratch, for callers that cannot
 * allocate device memory: for example code inside a host framework that
 * owns every device allocation and passes in only input and output
 * buffers, or latency-critical paths that forbid cudaMalloc because it can
 * synchronise the device.  The paper has no counterpart; this is a library
 * convenience.  Arguments and results are those of tadm_head_confidence.
 *  - The partials live in a fixed device array of
 *    TADM_HEAD_STATIC_SCRATCH_BYTES (8 MiB) inside the library, which every
 *    GPU that loads the library holds until the process exits.  Calls that
 *    need more than that (tadm_head_scratch_size) return
 *    TADM_ERR_INVALID_ARG and do nothing.
 *  - The first call on each device looks up the array's device address
 *    (cudaGetSymbolAddress, with that device current); make that first call
 *    before any stream capture.  Later calls on the device only launch.
 *    Like every entry point of this library it assumes one device per
 *    process whose context lives until exit: after cudaDeviceReset the
 *    remembered address is stale and the library must not be called again.
 *  - Argument errors are those of tadm_head_confidence, checked in the same
 *    order (also when rows == 0).
 *  - No allocation of any kind: no cudaMalloc / cudaFree, no allocating
 *    library routine.
 *  - Every call shares the one array and leaves its partials there; nothing
 *    in it needs to start at zero.  Calls whose work overlaps on the GPU
 *    (other streams, other host threads) race on the array: serialise them. */
#define TADM_HEAD_STATIC_SCRATCH_BYTES (8u << 20)
TADM_API tadm_status tadm_head_confidence_static(const void* x, const void* w, int rows, int d, int vocab,
                                                 int mask_id, int dtype, float* conf, int32_t* tok,
                                                 tadm_stream stream);

/* softmax(Q K^T / sqrt(hd)) V for queries at positions ctx .. ctx+rows-1 over
 * keys 0 .. ctx+rows-1 (keys < ctx always visible; the rest bidirectional,
 * or causal if `causal`).  window > 0 (a local layer): a query at position p
 * sees only keys j with p - j < window as well; 0 = no window.  dtype 1:
 * bf16, 0: fp32.
 * q: [batch, n_heads, rows, hd]; k: [batch, n_kv_heads, kv_stride, hd];
 * v transposed: [batch, n_kv_heads, hd, kv_stride]; o: [batch*rows, n_heads*hd].
 * K and V entries at positions >= ctx + rows must hold finite values. */
TADM_API tadm_status tadm_attention(const void* q, const void* k, const void* v, void* o, int batch,
                           int n_heads, int n_kv_heads, int head_dim, int rows, int ctx,
                           int kv_stride, int causal, int window, int dtype, tadm_stream stream);

/* ------------------------------------------------------------ ReMDM sampler --
 * The paper's Pretraining sampler in place of the confidence top-k: the
 * remasking reverse step of §5 Eq. (inf-post-TADM) (App. B Eqs.
 * remdm-posterior, remdm-param) with the fused prediction, nucleus (top-p)
 * sampling and the ReMDM-Cap / ReMDM-Loop schedules of App. C.2.  Readings
 * where the paper defers to ReMDM without restating it:
 *  - kind 0 (Cap): alpha_t = 1 - t on t = (T - n) / T; sigma_t = min(eta,
 *    sigma_max), sigma_max = min(1, (1 - alpha_s) / alpha_t);
 *  - kind 1 (Loop): alpha rises linearly to alpha_on at t_on, stays there
 *    to t_off, then rises to 1; sigma_t = min(eta, sigma_max) while alpha_t =
 *    alpha_s = alpha_on, else 0;
 *  - a generated token is remasked if u0 < sigma_t; a masked position takes a
 *    token if u1 < p_unmask = (alpha_s - (1 - sigma_t) alpha_t) / (1 - alpha_t);
 *    prompt positions never change;
 *  - the token: nucleus N = {v != MASK : q_v >= tau}, tau the largest value
 *    whose tokens hold >= top_p of the mass (ties kept); the first v of N in
 *    id order whose cumulative mass in N exceeds u2 * mass(N);
 *  - draws: Philox4x32-10 (Salmon et al., SC'11), counter (block lo, block
 *    hi, 0x52454D44, 0), key (seed lo, seed hi), block (step * batch + b) *
 *    rows + r for canvas position (b, r); u_j = (word j >> 8) * 2^-24. */

/* Host only: out = {alpha_t, alpha_s, sigma_t, p_unmask} of reverse step n
 * (0 .. T-1) of schedule `kind` (0 Cap, 1 Loop; t_on, t_off, alpha_on are
 * read by Loop only).  INVALID_ARG for T < 1, n outside 0..T-1, eta < 0, or
 * a Loop with 0 < t_off < t_on < 1 and 0 < alpha_on < 1 violated. */
TADM_API tadm_status tadm_remdm_schedule(int kind, int T, int n, double eta, double t_on, double t_off,
                                         double alpha_on, double out[4]);

/* The three draws of every canvas position at reverse step `step`:
 * out (device float [batch * rows * 3]) = (u0, u1, u2) per position in
 * row-major (b, r) order. */
TADM_API tadm_status tadm_remdm_uniforms(uint64_t seed, int step, int batch, int rows, float* out,
                                         tadm_stream stream);

/* One ReMDM reverse step on a canvas, from given logits.  z: device int32
 * [batch, rows] (leading dimension ldz), updated in place; logits: device
 * fp32 [batch * rows, vocab] (row stride ld_logits), row b * rows + r for
 * position (b, r), read only; positions < first_gen never change; sigma and
 * p_unmask as from tadm_remdm_schedule; action: device int32 [batch * rows],
 * written with 0 keep, 1 remask, 2 unmask.  No allocation. */
TADM_API tadm_status tadm_remdm_update(int32_t* z, int ldz, const float* logits, int ld_logits, int batch, int rows,
                                       int first_gen, int vocab, int mask_id, double sigma, double p_unmask,
                                       float top_p, uint64_t seed, int step, int32_t* action, tadm_stream stream);

/* Whole generation with the ReMDM sampler (single block: prompt + gen_len
 * masks): Alg. 1's refresh when n mod K == 0, the fused prediction every
 * step, then the ReMDM step of schedule `kind` (eta; Loop with t_on 0.55,
 * t_off 0.05, alpha_on 0.9 as in App. C.2).  logits_scratch: caller device
 * fp32 buffer of at least batch * gen_len * vocab * 4 bytes (the logits of
 * the masked rows of a step).  Positions still masked after the last step
 * cannot occur: the last step unmasks every masked position.  The handle
 * needs max_rows >= prompt_len + gen_len and no KV context. */
TADM_API tadm_status tadm_generate_remdm(tadm_handle* h, const int32_t* prompt, int batch, int prompt_len,
                                         int32_t* out, int gen_len, int steps, int K, int kind, double eta,
                                         float top_p, uint64_t seed, float* logits_scratch, size_t scratch_bytes,
                                         tadm_stream stream);

/* ---------------------------------------------------- entropy-bound sampler --
 * The paper's Post-training sampler (App. C.1 "Sampler Details", Alg. 2:
 * DiffusionGemma entropy-bound sampling) with Alg. 1's anchor cache.  Per
 * reverse step n = T .. 1 and generated position l:
 *  - tau_n = tau_min + (tau_max - tau_min) n / T; p = softmax(L / tau_n) over
 *    the ids != MASK (MASK = vocab - 1 gets p = 0); the argmax takes the
 *    lowest id among equal logits; H = -sum p log p;
 *  - n > 1: the draw from Cat(p) is the first id whose cumulative p exceeds
 *    u0 (id order); positions sorted by ascending H (ties to the lower
 *    position) with C_m the summed and M_m the largest entropy of the first
 *    m: pi_m keeps its draw when C_m - M_m <= eta, every other generated
 *    position takes the re-noise token floor(u1 (vocab - 1)); n = 1: every
 *    generated position takes its argmax;
 *  - self-conditioning: s = p E (E the embedding table) is added to the
 *    input embedding of the generated positions at the next step; s = 0 at
 *    n = T;
 *  - readings: the initial canvas z_T is the prompt followed by re-noise
 *    tokens of step T; refresh at step i = T - n when i mod K == 0; the
 *    anchor pass of a refresh step embeds the same canvas plus s;
 *  - draws: the ReMDM Philox stream above, (u0, u1, unused) of position
 *    (b, r) at step i = T - n, and step T for the initial canvas.
 * Arithmetic: fp32 logits, exponentials and sums; the accepted set from the
 * fp32 entropies with fp64 partial sums. */

/* One step of Alg. 2 from given logits.  z: device int32 [batch, rows]
 * (leading dimension ldz); the positions first_gen .. rows-1 (G = rows -
 * first_gen, 1 <= G <= 16384) are rewritten, the others never change.
 * logits: device fp32, row b * G + g (stride ld_logits) for position
 * (b, first_gen + g), read only.  tau > 0 is tau_n; last = 1 for n = 1
 * (argmax only; entropy, probs and eta unused), else 0.  entropy: device
 * fp32 [batch * G], written with H (n > 1).  probs (optional, may be NULL):
 * written with q = exp((L - max) / tau) (0 for MASK), row stride ld_probs,
 * fp32 (probs_dtype 0) or bf16 (1); z_sum (optional): fp32 [batch * G],
 * written with Z = sum q, so that p = q / Z.  No allocation; INVALID_ARG for
 * bad sizes, NaN eta or tau <= 0. */
TADM_API tadm_status tadm_eb_update(int32_t* z, int ldz, const float* logits, int ld_logits, int batch, int rows,
                                    int first_gen, int vocab, int mask_id, double tau, double eta, int last,
                                    uint64_t seed, int step, float* entropy, void* probs, int probs_dtype,
                                    int ld_probs, float* z_sum, tadm_stream stream);

/* Bytes of caller scratch that tadm_generate_entropy_bound needs: the
 * logits of the generated rows (fp32 [batch * gen_len, vocab]), with
 * self-conditioning q ([batch * gen_len, vocab]) and E^T ([d_model, vocab])
 * in the model's element type, q E (fp32 [batch * gen_len, d_model]) and Z
 * (fp32 [batch * gen_len]), and the entropies (fp32 [batch * gen_len]);
 * 256-byte aligned segments.  The self-conditioning signal s = p E is
 * applied as (q E) / Z in the next step's embedding. */
TADM_API tadm_status tadm_eb_scratch_bytes(const tadm_handle* h, int batch, int gen_len, int self_cond,
                                           size_t* bytes);

/* Whole generation with the entropy-bound sampler on one canvas (prompt +
 * gen_len generated positions, bidirectional; the handle needs max_rows >=
 * prompt_len + gen_len and no KV context): `steps` = T reverse steps,
 * anchor refresh every K, eta, tau_max >= tau_min > 0, self_cond 0/1.
 * scratch: device, 256-byte aligned, at least tadm_eb_scratch_bytes.
 * out: device int32 [batch, prompt_len + gen_len]. */
TADM_API tadm_status tadm_generate_entropy_bound(tadm_handle* h, const int32_t* prompt, int batch, int prompt_len,
                                                 int32_t* out, int gen_len, int steps, int K, double eta,
                                                 double tau_max, double tau_min, int self_cond, uint64_t seed,
                                                 void* scratch, size_t scratch_bytes, tadm_stream stream);

#ifdef __cplusplus
}
#endif
#endif /* TADM_H */
