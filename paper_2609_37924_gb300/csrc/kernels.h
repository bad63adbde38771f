// Host-side launchers of the sm_103a kernels (internal to libtadm).  Each
// returns nullptr on success or a static error string.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "epilogue.cuh"

namespace tadm {

// Launches with programmatic stream serialization (the kernel begins with
// pdl_enter()), unless the environment sets TADM_PDL=0.
bool pdl_enabled();
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl_enabled() ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

struct GemmCall {
  const void* A;   // [M, K] (A_rows rows visible to the tensor map when > 0)
  const void* B;   // [N, K]  (EPI_GLU: [2N, K], gate rows then up rows)
  int M, N, K, lda, ldb;
  int64_t A_rows;
  int epi;
  EpiParams ep;
  int* status;
  const int* m_dev = nullptr;   // optional device row count <= M (tcgen05 path): tiles past it are skipped
  int k_b = 0;           // > 0: B has k_b columns and A's K = 2 k_b columns [hi | lo] both multiply B (split operand)
  float* split_buf;      // fp32 partials for split-K (null: no split)
  size_t split_bytes;
  int launched;          // out: kernels launched
};

// Split-K partial buffer that covers every GEMM (units x 128 x 256 fp32 for at most one unit per SM).
size_t gemm_tc_split_bytes();

// tcgen05 path (bf16 operands)
const char* gemm_tc(const GemmCall& g, cudaStream_t s);
int gemm_tc_tiles_n(int N, int epi);
// fixed-order sum of split-K partials followed by the GEMM's epilogue; *launches = kernels it launched
const char* splitk_reduce(int epi, const EpiParams& ep, const float* part, size_t part_stride, int ldp, int splits,
                          int n_tiles_n, cudaStream_t s, int* launches);
// CUDA-core path (fp32 operands)
const char* gemm_simt(const GemmCall& g, cudaStream_t s);
int gemm_simt_tiles_n(int N, int epi);

// q [B, Hq, rows, hd]; k [B, Hkv, kv_stride, hd]; v transposed [B, Hkv, hd, kv_stride]
struct AttnCall {
  const void *q, *k, *v;
  void* o;
  int batch, n_heads, n_kv_heads, head_dim, rows, ctx, kv_stride, causal;
  int bf16;
  int* status;   // device status word (may be null)
  void* part = nullptr;      // optional fp32 scratch for split-key partials (16-byte aligned)
  size_t part_bytes = 0;
  int window = 0;            // > 0: a query at position p sees only keys j with p - j < window
};
const char* attention(const AttnCall& a, cudaStream_t s);

// row kernels (act = bf16 when act_bf16 else fp32)
// out (and out2) = E[z]; with `add`, rows r >= add_first of sequence b also add
// add[a * d ..] / add_div[a] (add_div optional), a = b * (rows - add_first) + r - add_first
// (the self-conditioning signal)
const char* embed_rows(const int32_t* z, int ldz, int batch, int rows, const void* E, int e_bf16, int d,
                       int vocab, float* out, float* out2, cudaStream_t s, const float* add = nullptr,
                       int add_first = 0, const float* add_div = nullptr);
// lo_off > 0 (bf16 activations): also the remainder bf16(y - bf16(y)) at column lo_off of each output row
const char* rmsnorm_rows(const float* x, int M, int d, const void* gain, int w_bf16, float eps, void* out,
                         int ldo, int act_bf16, cudaStream_t s, const int32_t* rows_idx = nullptr, int lo_off = 0);
// per sequence: the rows still holding MASK (first `per_seq` of them, in order) -> idx[b * per_seq + j]
// (global row b * rows + r); conf of every row set to -inf so that rows left out are never selected
const char* masked_rows(const int32_t* z, int ldz, int batch, int rows, int mask_id, int per_seq, int32_t* idx,
                        float* conf, cudaStream_t s);
const char* ln_pair_rows(const float* c, const float* h, int M, int d, const void* wc, const void* bc,
                         const void* wh, const void* bh, int w_bf16, float eps, void* u, int act_bf16,
                         cudaStream_t s);
const char* layernorm_rows(const float* x, int M, int d, const void* w, const void* b, int w_bf16, float eps,
                           float* out, cudaStream_t s);
const char* rms_scale_rows(const float* x, int M, int d, float eps, float* s_out, cudaStream_t st);
// sandwich norm: x += y / sqrt(mean(y^2) + eps) * g_post; with g_next, also
// out = x / sqrt(mean(x^2) + eps) * g_next (the next sub-block's pre-norm, act type)
const char* post_norm_add(float* x, const float* y, int M, int d, const void* g_post, const void* g_next, int w_bf16,
                          float eps, void* out, int act_bf16, cudaStream_t s);
const char* scale_rows(const float* x, const float* sc, int M, int d, void* out, int act_bf16, cudaStream_t s);
const char* concat_rows(const float* const* parts, const int* widths, int n_parts, int M, void* out,
                        int act_bf16, cudaStream_t s);
const char* sub_rows(const float* a, const float* b, int M, int d, float* out, cudaStream_t s);
const char* rope_table(float2* tab, int n_pos, int head_dim, float theta, cudaStream_t s);
const char* fill_canvas(int32_t* z, int ldz, const int32_t* prompt, int batch, int prompt_len, int total,
                        int mask_id, cudaStream_t s);
const char* copy_rows_i32(const int32_t* src, int lds, int32_t* dst, int ldd, int batch, int cols,
                          cudaStream_t s);

// sampler
const char* confidence_rows(const float* logits, int rows, int vocab, int ld, int mask_id, float* conf,
                            int32_t* tok, cudaStream_t s);
const char* combine_partials(const float* part, int rows, int n_tiles, float* conf, int32_t* tok,
                             cudaStream_t s, const int32_t* rows_idx = nullptr);
// ReMDM sampler: the draws of a step; decide (and apply remasks); nucleus tokens of the unmasking rows
const char* remdm_uniforms(uint64_t seed, int step, int B, int R, float* out, cudaStream_t s);
const char* remdm_decide(int32_t* z, int ldz, int B, int R, int first_gen, int mask_id, double sigma,
                         double p_unmask, uint64_t seed, int step, int32_t* act, cudaStream_t s);
const char* remdm_sample(const float* logits, int ld, int n_rows, const int32_t* idx, const int32_t* act, int32_t* z,
                         int ldz, int B, int R, int vocab, int mask_id, float top_p, uint64_t seed, int step,
                         cudaStream_t s, const int* count = nullptr);
// rows with action 2 in row order into idx[0 .. *count), padded to `bound` entries
const char* remdm_rows(const int32_t* act, int n, int bound, int32_t* idx, int* count, cudaStream_t s);
const char* topk_unmask(int32_t* z, int ldz, const float* conf, const int32_t* tok, int batch, int rows, int k,
                        int mask_id, int32_t* selected, cudaStream_t s);
// entropy-bound sampler (Alg. 2): the generated positions first .. R-1 of each sequence
const char* eb_noise(int32_t* z, int ldz, int B, int R, int first, int vocab, uint64_t seed, int step, cudaStream_t s);
const char* eb_rows(int32_t* idx, int B, int R, int first, cudaStream_t s);
// part (optional): the output head's [rows][n_tiles][3] partials of these logits (max and argmax from them);
// q (optional): exp((l - max) / tau) per id; H: entropies; Zs (optional): Z = sum q per row
const char* eb_row(const float* logits, int ld, int B, int R, int first, int32_t* z, int ldz, int vocab, int mask_id,
                   float inv_tau, int last, uint64_t seed, int step, const float* part, int n_tiles, void* q,
                   int q_bf16, int ldq, float* H, float* Zs, cudaStream_t s);
int eb_max_gen();
const char* eb_accept(const float* H, int B, int R, int first, int32_t* z, int ldz, int vocab, double eta,
                      uint64_t seed, int step, cudaStream_t s);
// out [cols, rows] = in [rows, cols]^T (bf16: 2-byte elements, else fp32)
const char* transpose(const void* in, int rows, int cols, int bf16, void* out, cudaStream_t s);

}  // namespace tadm
