// libtadm: C ABI, model graph and the anchor-cache scheduler (Alg. 1).
//
// Host code only: every step of the path runs in the kernels of gemm_tc.cu /
// gemm_simt.cu, attention.cu, rowops.cu and sampler.cu.  The library owns no
// device memory; the caller binds one workspace that is carved into the
// activation buffers, the per-layer KV caches of block mode, the internal
// anchor cache of tadm_generate, the RoPE table and the status word.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/tadm.h"
#include "kernels.h"

using namespace tadm;

namespace {

struct LayerW {
  const void *attn_norm, *wqkv, *wo, *ffn_norm, *wgu, *wdown;
  const void *q_norm, *k_norm, *post_attn, *post_ffn;   // Gemma-3 details (null when off)
  int window;      // > 0: local layer with this sliding window
  int global;      // 1: global layer (RoPE base rope_theta_global when set)
};

struct Inventory {
  std::vector<std::string> names;
  std::vector<int64_t> rows, cols;
};

bool valid_config(const tadm_config* c, std::string* why) {
  auto fail = [&](const char* m) {
    if (why) *why = m;
    return false;
  };
  if (!c) return fail("config is NULL");
  if (c->vocab < 2 || c->d_model <= 0 || c->n_heads <= 0 || c->n_kv_heads <= 0 || c->head_dim <= 0 || c->ffn <= 0)
    return fail("sizes must be positive (vocab >= 2)");
  if (c->n_heads % c->n_kv_heads) return fail("n_heads must be a multiple of n_kv_heads");
  if (c->head_dim % 2) return fail("head_dim must be even");
  if (c->glu != 0 && c->glu != 1) return fail("glu must be 0 or 1");
  if (c->n_shared < 0 || c->n_anchor < 0 || c->n_denoise < 0) return fail("layer counts must be >= 0");
  if (c->fusion < 0 || c->fusion > 2) return fail("fusion must be 0, 1 or 2");
  if (c->fusion == 1 && (c->fusion_rank <= 0 || c->fusion_heads <= 0 || c->fusion_rank % c->fusion_heads))
    return fail("fusion_rank must be a positive multiple of fusion_heads");
  if (c->dtype != 0 && c->dtype != 1) return fail("dtype must be 0 (fp32) or 1 (bf16)");
  if (!(c->norm_eps >= 0.0f) || !(c->rope_theta > 0.0f)) return fail("norm_eps >= 0 and rope_theta > 0");
  if (c->sliding_window < 0 || c->global_every < 0) return fail("sliding_window and global_every must be >= 0");
  if ((c->qk_norm != 0 && c->qk_norm != 1) || (c->sandwich_norm != 0 && c->sandwich_norm != 1))
    return fail("qk_norm and sandwich_norm must be 0 or 1");
  if (c->qkv_split != 0 && c->qkv_split != 1) return fail("qkv_split must be 0 or 1");
  if (!(c->rope_theta_global >= 0.0f)) return fail("rope_theta_global must be >= 0");
  return true;
}

Inventory inventory(const tadm_config* c) {
  Inventory inv;
  auto add = [&](const std::string& n, int64_t r, int64_t k) {
    inv.names.push_back(n);
    inv.rows.push_back(r);
    inv.cols.push_back(k);
  };
  const int64_t d = c->d_model, hd = c->head_dim, F = c->ffn;
  add("embed", c->vocab, d);
  const char* nets[3] = {"shared", "anchor", "denoise"};
  const int counts[3] = {c->n_shared, c->n_anchor, c->n_denoise};
  for (int t = 0; t < 3; ++t)
    for (int i = 0; i < counts[t]; ++i) {
      std::string p = std::string(nets[t]) + "." + std::to_string(i) + ".";
      add(p + "attn_norm", d, 1);
      add(p + "wqkv", (c->n_heads + 2LL * c->n_kv_heads) * hd, d);
      if (c->qk_norm) {
        add(p + "q_norm", hd, 1);
        add(p + "k_norm", hd, 1);
      }
      add(p + "wo", d, c->n_heads * hd);
      if (c->sandwich_norm) add(p + "post_attn_norm", d, 1);
      add(p + "ffn_norm", d, 1);
      add(p + "wgu", 2 * F, d);
      add(p + "wdown", d, F);
      if (c->sandwich_norm) add(p + "post_ffn_norm", d, 1);
    }
  if (c->fusion == 0) {
    add("fusion.ln_c.w", d, 1);
    add("fusion.ln_c.b", d, 1);
    add("fusion.ln_h.w", d, 1);
    add("fusion.ln_h.b", d, 1);
    add("fusion.w_g1", 5 * d, 2 * d);
    add("fusion.b_g1", 5 * d, 1);
    add("fusion.w2", d, 4 * d);
    add("fusion.b2", d, 1);
    add("fusion.ln_out.w", d, 1);
    add("fusion.ln_out.b", d, 1);
  } else if (c->fusion == 1) {
    const int64_t r = c->fusion_rank;
    add("fusion.wc", r, d);
    add("fusion.wh", r, d);
    add("fusion.wqkv", 3 * r, 2 * r);
    add("fusion.wo", r, r);
    add("fusion.w1", 2 * r, r);
    add("fusion.w2", r, 2 * r);
    add("fusion.wg1", r, 4 * r);
    add("fusion.wg2", 1, r);
    add("fusion.bg", 1, 1);
    add("fusion.wup", d, r);
  }
  add("final_norm", d, 1);
  if (!c->tied_lm_head) add("lm_head", c->vocab, d);
  return inv;
}

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace

struct tadm_handle {
  tadm_config cfg{};
  Inventory inv;
  std::vector<const void*> w;
  int max_batch = 0, max_rows = 0, max_ctx = 0;
  int L_total = 0;
  std::vector<LayerW> layers;
  const void *embed = nullptr, *final_norm = nullptr, *lm_head = nullptr;
  // fusion parameters, indexed by inventory name
  const void* fw[12] = {};

  // workspace
  char* ws = nullptr;
  size_t ws_bytes = 0, ws_need = 0;
  struct Off {
    size_t status, rope, rope_g, post, c, x, h_int, norm, qbuf, kv, attn, glu, f_g, f_hid, f_pre, part, conf, tok,
        split, idx;
    size_t attn_part, act, cnt;
    size_t pa_z, pa_j, pa_mq, pa_mk, pa_mv, pa_mo, pa_r, pa_rb, pa_hid, pa_phi, pa_m, pa_dz, pa_f, pa_g, pa_mb;
  } off{};
  size_t kv_slab = 0;
  int kv_stride = 0, n_part_tiles = 0;

  // GEMM timing probe
  std::vector<cudaEvent_t> probe_ev;
  std::vector<double> probe_flops, probe_bytes;   // algorithmic FLOPs and bytes of each record
  std::vector<int> probe_kind;
  int probe_next = 0;

  // sequence state
  int batch = 0, ctx = 0;
  tadm_counters counters{};
  cudaStream_t last_stream = nullptr;
  std::string err;

  // CUDA graph of a repeated tadm_generate call (same sizes and pointers,
  // workspace included): the second such call is captured on an internal
  // stream, later ones replay it.  The host-side results of the captured run
  // (counters, context length) are restored on replay.  Binding a workspace
  // destroys the graph.
  cudaStream_t gstream = nullptr;
  cudaEvent_t gev_in = nullptr, gev_out = nullptr;
  cudaGraphExec_t gexec = nullptr;
  int64_t gkey[9] = {}, gkey_seen[9] = {};   // sizes, prompt, out and workspace pointers
  tadm_counters gcounters{};
  int gctx = 0;

  int es() const { return cfg.dtype ? 2 : 4; }
  bool has_rope_g() const {
    if (!(cfg.rope_theta_global > 0.0f) || cfg.rope_theta_global == cfg.rope_theta) return false;
    for (const auto& L : layers)
      if (L.global) return true;
    return false;
  }
  int act_bf16() const { return cfg.dtype; }
  template <class T = char>
  T* at(size_t o) const { return reinterpret_cast<T*>(ws + o); }
  int* status() const { return at<int>(off.status); }
};

namespace {

tadm_status fail(tadm_handle* h, tadm_status s, const char* fmt, ...) {
  if (h) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    h->err = buf;
  }
  return s;
}

#define TRY(expr)                                                   \
  do {                                                              \
    const char* _e = (expr);                                        \
    if (_e) return fail(h, TADM_ERR_CUDA, "%s: %s", #expr, _e);     \
    h->counters.kernel_launches += 1;                               \
  } while (0)

#define TRYS(expr)                         \
  do {                                     \
    tadm_status _s = (expr);               \
    if (_s != TADM_OK) return _s;          \
  } while (0)

// fp32 scratch for the split-key partials of attention (bf16 models)
constexpr size_t kAttnPartBytes = size_t(64) << 20;

size_t cache_bytes(const tadm_config& c, int batch, int rows) {
  const size_t M = static_cast<size_t>(batch) * rows;
  if (c.fusion != 1) return align_up(M * c.d_model * 4, 256);   // h only (fusion 0 and 2)
  const size_t r = c.fusion_rank;
  // H0 [M,d] | sC [M] | sH [M] | Z0 [M,r] | U [M,r] | phi0 [M,r]   (fp32)
  return align_up(M * c.d_model * 4, 256) + 2 * align_up(M * 4, 256) + 3 * align_up(M * r * 4, 256);
}

struct CacheView {
  float *h, *sC, *sH, *Z0, *U, *phi0;
};
CacheView cache_view(const tadm_config& c, void* base, int batch, int rows) {
  CacheView v{};
  const size_t M = static_cast<size_t>(batch) * rows;
  char* p = static_cast<char*>(base);
  v.h = reinterpret_cast<float*>(p);
  if (c.fusion != 1) return v;
  const size_t r = c.fusion_rank;
  p += align_up(M * c.d_model * 4, 256);
  v.sC = reinterpret_cast<float*>(p);
  p += align_up(M * 4, 256);
  v.sH = reinterpret_cast<float*>(p);
  p += align_up(M * 4, 256);
  v.Z0 = reinterpret_cast<float*>(p);
  p += align_up(M * r * 4, 256);
  v.U = reinterpret_cast<float*>(p);
  p += align_up(M * r * 4, 256);
  v.phi0 = reinterpret_cast<float*>(p);
  return v;
}

void layout(tadm_handle* h) {
  const tadm_config& c = h->cfg;
  const size_t M = static_cast<size_t>(h->max_batch) * h->max_rows;
  const size_t d = c.d_model, es = h->es();
  const size_t q = static_cast<size_t>(c.n_heads) * c.head_dim;
  const size_t kv = static_cast<size_t>(c.n_kv_heads) * c.head_dim;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o = align_up(o + bytes, 256);
    return at;
  };
  h->kv_stride = static_cast<int>(align_up(static_cast<size_t>(h->max_ctx > 0 ? h->max_ctx : h->max_rows), 8));
  const int n_pos = h->kv_stride + h->max_rows;
  h->n_part_tiles = c.dtype ? gemm_tc_tiles_n(c.vocab, EPI_LMHEAD) : gemm_simt_tiles_n(c.vocab, EPI_LMHEAD);
  auto& f = h->off;
  f.status = take(256);
  f.rope = take(static_cast<size_t>(n_pos) * (c.head_dim / 2) * 8);
  // global layers with their own RoPE base get a second table
  f.rope_g = h->has_rope_g() ? take(static_cast<size_t>(n_pos) * (c.head_dim / 2) * 8) : f.rope;
  f.post = c.sandwich_norm ? take(M * d * 4) : 0;   // sub-block output ahead of its post-norm
  f.c = take(M * d * 4);
  f.x = take(M * d * 4);
  f.h_int = take(cache_bytes(c, h->max_batch, h->max_rows));
  f.norm = take(M * 2 * d * es);
  f.qbuf = take(M * q * es);
  h->kv_slab = align_up(static_cast<size_t>(h->max_batch) * kv * h->kv_stride * es, 256);
  const int n_kv_layers = h->max_ctx > 0 ? h->L_total : 1;
  f.kv = take(h->kv_slab * 2 * (n_kv_layers > 0 ? n_kv_layers : 1));
  f.attn = take(M * q * es);
  f.glu = take(M * c.ffn * es);
  if (c.fusion == 0) {
    f.f_g = take(M * d * es);
    f.f_hid = take(M * 4 * d * es);
    f.f_pre = take(M * d * 4);
  } else if (c.fusion == 1) {
    const size_t r = c.fusion_rank;
    f.pa_z = take(M * r * 4);
    f.pa_j = take(M * 4 * r * es);
    f.pa_mq = take(M * r * es);
    f.pa_mk = take(M * r * es);
    f.pa_mv = take(M * r * es);
    f.pa_mo = take(M * r * es);
    f.pa_r = take(M * r * 4);
    f.pa_rb = take(M * r * es);
    f.pa_hid = take(M * 2 * r * es);
    f.pa_phi = take(M * r * 4);
    f.pa_m = take(M * r * 4);
    f.pa_dz = take(M * r * 4);
    f.pa_f = take(M * 4 * r * es);
    f.pa_g = take(M * 4);
    f.pa_mb = take(M * r * es);
  }
  f.part = take(M * h->n_part_tiles * 3 * 4);
  f.split = c.dtype ? take(gemm_tc_split_bytes()) : take(0);
  f.attn_part = c.dtype ? take(kAttnPartBytes) : take(0);
  f.act = take(M * 4);       // ReMDM: per-position actions
  f.cnt = take(256);         // ReMDM: device count of unmasking rows
  f.conf = take(M * 4);
  f.tok = take(M * 4);
  f.idx = take(M * 4);
  h->ws_need = o;
}

// --------------------------------------------------------------------------- kernels wrappers
// probe kinds beyond the GEMM epilogues (0..10)
constexpr int kProbeAttention = 11, kProbeNorm = 12, kProbeAttentionShort = 13;   // 13: attention of < 128 rows
// Opens a probe record (start event) when the probe is on and has room: returns its index, else -1.
int probe_begin(tadm_handle* h, cudaStream_t s) {
  if (h->probe_next >= static_cast<int>(h->probe_flops.size())) return -1;
  cudaEventRecord(h->probe_ev[2 * h->probe_next], s);
  return h->probe_next++;
}
void probe_end(tadm_handle* h, cudaStream_t s, int idx, int kind, double flops, double bytes = 0.0) {
  if (idx < 0) return;
  cudaEventRecord(h->probe_ev[2 * idx + 1], s);
  h->probe_kind[idx] = kind;
  h->probe_flops[idx] = flops;
  h->probe_bytes[idx] = bytes;
}

// k_b > 0: A = [hi | lo] holds 2 k_b columns (a split operand) and both halves multiply B's k_b columns;
// the recorded work is that of the k_b-deep product the method computes.
tadm_status gemm(tadm_handle* h, const void* A, int64_t a_rows, int lda, const void* B, int ldb, int M, int N, int K,
                 int epi, const EpiParams& ep, cudaStream_t s, bool out_f32 = false, const int* m_dev = nullptr,
                 int k_b = 0) {
  GemmCall g{};
  g.k_b = k_b;
  g.A = A;
  g.B = B;
  g.M = M;
  g.N = N;
  g.K = K;
  g.lda = lda;
  g.ldb = ldb;
  g.A_rows = a_rows;
  g.epi = epi;
  g.ep = ep;
  g.status = h->status();
  g.m_dev = m_dev;
  if (h->cfg.dtype) {
    g.split_buf = h->at<float>(h->off.split);
    g.split_bytes = gemm_tc_split_bytes();
  }
  g.ep.out_bf16 = out_f32 ? 0 : h->act_bf16();
  g.ep.bias_bf16 = h->cfg.dtype;
  const int pi = probe_begin(h, s);
  const char* e = h->cfg.dtype ? gemm_tc(g, s) : gemm_simt(g, s);
  if (e) return fail(h, TADM_ERR_CUDA, "GEMM (M=%d N=%d K=%d epi=%d): %s", M, N, K, epi, e);
  h->counters.kernel_launches += h->cfg.dtype ? g.launched : 1;
  const double n_acc = epi == EPI_GLU ? 2.0 * N : static_cast<double>(N);
  if (k_b > 0) K = k_b;
  // algorithmic bytes: A and B read once, the output written once (fp32 or
  // the activation type), the residual stream read and written by EPI_RESID
  const double es = h->es(), out_es = (epi == EPI_RESID || out_f32 || !h->act_bf16()) ? 4.0 : es;
  const double bytes = es * (static_cast<double>(M) * K + n_acc * K) + out_es * M * N +
                       (epi == EPI_RESID ? 4.0 * M * N : 0.0);
  probe_end(h, s, pi, epi, 2.0 * M * n_acc * K, epi == EPI_LMHEAD ? es * (static_cast<double>(M) * K + n_acc * K)
                                                                  : bytes);
  return TADM_OK;
}

void* kv_ptr(tadm_handle* h, int li, int which) {
  const int slot = h->max_ctx > 0 ? li : 0;
  return h->at(h->off.kv + h->kv_slab * (2 * slot + which));
}

// Pre-norm backbone layer on the fp32 residual x [B*R, d], rows at positions
// ctx .. ctx+R-1, attending to the layer's KV context 0 .. ctx-1.  With the
// Gemma-3 details: QK-norm inside the QKV epilogue (before RoPE), the layer's
// window and RoPE table, and sandwich norms: the O and down projections then
// write their output to the post buffer, and one row kernel applies the
// post-norm and the residual add (after attention also the FFN pre-norm).
tadm_status layer_fwd(tadm_handle* h, int li, float* x, int B, int R, int ctx, int causal, cudaStream_t s) {
  const tadm_config& c = h->cfg;
  const LayerW& L = h->layers[li];
  const int M = B * R, d = c.d_model, hd = c.head_dim;
  const int q = c.n_heads * hd, nqkv = (c.n_heads + 2 * c.n_kv_heads) * hd;
  const int64_t Mmax = static_cast<int64_t>(h->max_batch) * h->max_rows;
  void* norm = h->at(h->off.norm);
  // qkv_split: the QKV projection's input enters the tensor cores as bf16 hi + lo (about 16 bits)
  const bool split = c.dtype && c.qkv_split;
  int pi = probe_begin(h, s);
  TRY(rmsnorm_rows(x, M, d, L.attn_norm, c.dtype, c.norm_eps, norm, split ? 2 * d : d, h->act_bf16(), s, nullptr,
                   split ? d : 0));
  probe_end(h, s, pi, kProbeNorm, 0.0);
  EpiParams ep{};
  ep.q = h->at(h->off.qbuf);
  ep.k = kv_ptr(h, li, 0);
  ep.v = kv_ptr(h, li, 1);
  ep.R = R;
  ep.ctx = ctx;
  ep.kv_stride = h->kv_stride;
  ep.n_heads = c.n_heads;
  ep.n_kv_heads = c.n_kv_heads;
  ep.head_dim = hd;
  ep.rope = 1;
  ep.rope_tab = h->at<const float2>(L.global ? h->off.rope_g : h->off.rope);
  ep.rope_npos = h->kv_stride + h->max_rows;
  ep.q_gain = L.q_norm;
  ep.k_gain = L.k_norm;
  ep.qk_eps = c.norm_eps;
  TRYS(gemm(h, norm, Mmax, split ? 2 * d : d, L.wqkv, d, M, nqkv, split ? 2 * d : d, EPI_QKV, ep, s, false, nullptr,
            split ? d : 0));
  AttnCall a{ep.q, ep.k, ep.v, h->at(h->off.attn), B, c.n_heads, c.n_kv_heads, hd, R, ctx, h->kv_stride, causal,
             h->act_bf16(), h->status()};
  a.window = L.window;
  if (c.dtype) {
    a.part = h->at(h->off.attn_part);
    a.part_bytes = kAttnPartBytes;
  }
  pi = probe_begin(h, s);
  TRY(attention(a, s));
  // keys seen per query row: all of them, or the causal average (window: at most the window)
  double keys = causal ? ctx + 0.5 * (R + 1) : static_cast<double>(ctx + R);
  if (L.window > 0) keys = std::min(keys, static_cast<double>(L.window + (causal ? 0 : R)));
  probe_end(h, s, pi, R < 128 ? kProbeAttentionShort : kProbeAttention, 4.0 * M * c.n_heads * keys * hd);
  EpiParams er{};
  er.resid = x;
  er.ldr = d;
  EpiParams ey{};                       // sandwich: the sub-block output, fp32, ahead of its post-norm
  ey.out = h->at(h->off.post);
  ey.ldo = d;
  float* post = h->at<float>(h->off.post);
  if (c.sandwich_norm) {
    TRYS(gemm(h, h->at(h->off.attn), Mmax, q, L.wo, q, M, d, q, EPI_STORE, ey, s, true));
    // x += RMSNorm(o W_o^T) * post_attn; norm = RMSNorm(x) * ffn_norm
    pi = probe_begin(h, s);
    TRY(post_norm_add(x, post, M, d, L.post_attn, L.ffn_norm, c.dtype, c.norm_eps, norm, h->act_bf16(), s));
    probe_end(h, s, pi, kProbeNorm, 0.0);
  } else {
    TRYS(gemm(h, h->at(h->off.attn), Mmax, q, L.wo, q, M, d, q, EPI_RESID, er, s));
    pi = probe_begin(h, s);
    TRY(rmsnorm_rows(x, M, d, L.ffn_norm, c.dtype, c.norm_eps, norm, d, h->act_bf16(), s));
    probe_end(h, s, pi, kProbeNorm, 0.0);
  }
  EpiParams eg{};
  eg.out = h->at(h->off.glu);
  eg.ldo = c.ffn;
  eg.glu = c.glu;
  TRYS(gemm(h, norm, Mmax, d, L.wgu, d, M, c.ffn, d, EPI_GLU, eg, s));
  if (c.sandwich_norm) {
    TRYS(gemm(h, h->at(h->off.glu), Mmax, c.ffn, L.wdown, c.ffn, M, d, c.ffn, EPI_STORE, ey, s, true));
    pi = probe_begin(h, s);
    TRY(post_norm_add(x, post, M, d, L.post_ffn, nullptr, c.dtype, c.norm_eps, nullptr, h->act_bf16(), s));
    probe_end(h, s, pi, kProbeNorm, 0.0);
  } else {
    TRYS(gemm(h, h->at(h->off.glu), Mmax, c.ffn, L.wdown, c.ffn, M, d, c.ffn, EPI_RESID, er, s));
  }
  return TADM_OK;
}

tadm_status stack_fwd(tadm_handle* h, int first, int n, float* x, int B, int R, int ctx, int causal, cudaStream_t s) {
  for (int i = 0; i < n; ++i) TRYS(layer_fwd(h, first + i, x, B, R, ctx, causal, s));
  return TADM_OK;
}

// S: c = embed(z) then L_S layers (c lives in the workspace).
// `add` (optional): the self-conditioning signal of rows add_first .. R-1 of
// each sequence, fp32 [B * (R - add_first), d], added to their embedding
// (divided by add_div[row] when add_div is given).
tadm_status run_S(tadm_handle* h, const int32_t* z, int ldz, int B, int R, int causal, cudaStream_t s,
                  const float* add = nullptr, int add_first = 0, const float* add_div = nullptr) {
  const tadm_config& c = h->cfg;
  float* cbuf = h->at<float>(h->off.c);
  TRY(embed_rows(z, ldz, B, R, h->embed, c.dtype, c.d_model, c.vocab, cbuf, nullptr, s, add, add_first, add_div));
  return stack_fwd(h, 0, c.n_shared, cbuf, B, R, h->ctx, causal, s);
}

// Mixer phi(Z, U) of the paired-attention fusion (App. C.1); writes phi (fp32 [M, r]).
tadm_status mixer(tadm_handle* h, const float* Z, const float* U, int B, int R, float* phi, cudaStream_t s) {
  const tadm_config& c = h->cfg;
  const int M = B * R, r = c.fusion_rank, fh = c.fusion_heads, hd = r / fh;
  const int64_t Mmax = static_cast<int64_t>(h->max_batch) * h->max_rows;
  const float* parts[2] = {Z, U};
  const int widths[2] = {r, r};
  void* J = h->at(h->off.pa_j);
  TRY(concat_rows(parts, widths, 2, M, J, h->act_bf16(), s));
  EpiParams eq{};
  eq.q = h->at(h->off.pa_mq);
  eq.k = h->at(h->off.pa_mk);
  eq.v = h->at(h->off.pa_mv);
  eq.R = R;
  eq.ctx = 0;
  eq.kv_stride = R;
  eq.n_heads = fh;
  eq.n_kv_heads = fh;
  eq.head_dim = hd;
  eq.rope = 0;
  TRYS(gemm(h, J, Mmax, 2 * r, h->fw[2], 2 * r, M, 3 * r, 2 * r, EPI_QKV, eq, s));
  AttnCall a{eq.q, eq.k, eq.v, h->at(h->off.pa_mo), B, fh, fh, hd, R, 0, R, 0, h->act_bf16(), h->status()};
  TRY(attention(a, s));
  EpiParams e1{};
  e1.base = Z;
  e1.ldb = r;
  e1.out = h->at(h->off.pa_r);
  e1.ldo = r;
  e1.out2 = h->at(h->off.pa_rb);
  e1.ldo2 = r;
  TRYS(gemm(h, h->at(h->off.pa_mo), Mmax, r, h->fw[3], r, M, r, r, EPI_ADD, e1, s));
  // EPI_ADD writes fp32 to out; out_bf16 only affects out2 (act copy)
  EpiParams e2{};
  e2.out = h->at(h->off.pa_hid);
  e2.ldo = 2 * r;
  TRYS(gemm(h, h->at(h->off.pa_rb), Mmax, r, h->fw[4], r, M, 2 * r, r, EPI_SILU, e2, s));
  EpiParams e3{};
  e3.base = h->at<float>(h->off.pa_r);
  e3.ldb = r;
  e3.out = phi;
  e3.ldo = r;
  TRYS(gemm(h, h->at(h->off.pa_hid), Mmax, 2 * r, h->fw[5], 2 * r, M, r, 2 * r, EPI_ADD, e3, s));
  return TADM_OK;
}

// Z = (X / s) W^T as fp32 [M, r]; X / s is staged in the norm buffer.
tadm_status project_scaled(tadm_handle* h, const float* X, const float* sc, const void* W, int M, float* Z,
                           cudaStream_t s) {
  const tadm_config& c = h->cfg;
  const int64_t Mmax = static_cast<int64_t>(h->max_batch) * h->max_rows;
  void* norm = h->at(h->off.norm);
  TRY(scale_rows(X, sc, M, c.d_model, norm, h->act_bf16(), s));
  EpiParams e{};
  e.out = Z;
  e.ldo = c.fusion_rank;
  return gemm(h, norm, Mmax, c.d_model, W, c.d_model, M, c.fusion_rank, c.d_model, EPI_STORE, e, s, true);
}

// A: h = A(c) into the cache (plus the refresh-only quantities of App. C.1).
tadm_status run_A(tadm_handle* h, int B, int R, int causal, void* cache, cudaStream_t s) {
  const tadm_config& c = h->cfg;
  const int M = B * R;
  CacheView cv = cache_view(c, cache, B, R);
  const float* cbuf = h->at<float>(h->off.c);
  if (cudaMemcpyAsync(cv.h, cbuf, static_cast<size_t>(M) * c.d_model * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "copy c -> h failed");
  TRYS(stack_fwd(h, c.n_shared, c.n_anchor, cv.h, B, R, h->ctx, causal, s));
  if (c.fusion == 1) {
    // s_C, s_H, Z0 = (C0/s_C) W_C, U = (H0/s_H) W_H, phi(Z0, U)
    TRY(rms_scale_rows(cbuf, M, c.d_model, 1e-6f, cv.sC, s));
    TRY(rms_scale_rows(cv.h, M, c.d_model, 1e-6f, cv.sH, s));
    TRYS(project_scaled(h, cbuf, cv.sC, h->fw[0], M, cv.Z0, s));
    TRYS(project_scaled(h, cv.h, cv.sH, h->fw[1], M, cv.U, s));
    TRYS(mixer(h, cv.Z0, cv.U, B, R, cv.phi0, s));
  }
  return TADM_OK;
}

// Phi: x = h~ = Phi(c, cache) (fp32 [M, d] in the workspace).
tadm_status run_fusion(tadm_handle* h, int B, int R, const void* cache, cudaStream_t s) {
  const tadm_config& c = h->cfg;
  const int M = B * R, d = c.d_model;
  const int64_t Mmax = static_cast<int64_t>(h->max_batch) * h->max_rows;
  CacheView cv = cache_view(c, const_cast<void*>(cache), B, R);
  const float* cbuf = h->at<float>(h->off.c);
  float* x = h->at<float>(h->off.x);
  if (c.fusion == 2) {
    // fusion off (the naive stale-anchor reuse of App. D): D reads h' itself
    if (cudaMemcpyAsync(x, cv.h, static_cast<size_t>(M) * d * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
      return fail(h, TADM_ERR_CUDA, "copy h -> x failed");
    return TADM_OK;
  }
  if (c.fusion == 0) {
    // u = [LN(c); LN(h)];  [g | a] = [sigmoid(W_g u + b_g) | GELU(W_1 u + b_1)];
    // pre = h + g * (W_2 a + b_2);  h~ = LN(pre)                        (App. C.2)
    void* u = h->at(h->off.norm);
    int pi = probe_begin(h, s);
    TRY(ln_pair_rows(cbuf, cv.h, M, d, h->fw[0], h->fw[1], h->fw[2], h->fw[3], c.dtype, c.norm_eps, u,
                     h->act_bf16(), s));
    probe_end(h, s, pi, kProbeNorm, 0.0);
    EpiParams e1{};
    e1.bias = h->fw[5];
    e1.d_split = d;
    e1.out = h->at(h->off.f_g);
    e1.ldo = d;
    e1.out2 = h->at(h->off.f_hid);
    e1.ldo2 = 4 * d;
    TRYS(gemm(h, u, Mmax, 2 * d, h->fw[4], 2 * d, M, 5 * d, 2 * d, EPI_FUSION1, e1, s));
    EpiParams e2{};
    e2.base = cv.h;
    e2.ldb = d;
    e2.gate = h->at(h->off.f_g);
    e2.ldg = d;
    e2.bias = h->fw[7];
    e2.out = h->at(h->off.f_pre);
    e2.ldo = d;
    TRYS(gemm(h, h->at(h->off.f_hid), Mmax, 4 * d, h->fw[6], 4 * d, M, d, 4 * d, EPI_FUSION2, e2, s));
    pi = probe_begin(h, s);
    TRY(layernorm_rows(h->at<float>(h->off.f_pre), M, d, h->fw[8], h->fw[9], c.dtype, c.norm_eps, x, s));
    probe_end(h, s, pi, kProbeNorm, 0.0);
    return TADM_OK;
  }
  // paired attention (App. C.1): Z = (C/s_C) W_C; M = phi(Z, U) - phi(Z0, U);
  // F = [U; Z0; Z - Z0; M]; g = sigmoid(SiLU(F W_g1) W_g2 + b_g); H~ = H0 + g s_H (M W_up)
  const int r = c.fusion_rank;
  float* Z = h->at<float>(h->off.pa_z);
  TRYS(project_scaled(h, cbuf, cv.sC, h->fw[0], M, Z, s));
  float* phi = h->at<float>(h->off.pa_phi);
  TRYS(mixer(h, Z, cv.U, B, R, phi, s));
  float* Mm = h->at<float>(h->off.pa_m);
  float* dZ = h->at<float>(h->off.pa_dz);
  TRY(sub_rows(phi, cv.phi0, M, r, Mm, s));
  TRY(sub_rows(Z, cv.Z0, M, r, dZ, s));
  const float* parts[4] = {cv.U, cv.Z0, dZ, Mm};
  const int widths[4] = {r, r, r, r};
  void* F = h->at(h->off.pa_f);
  TRY(concat_rows(parts, widths, 4, M, F, h->act_bf16(), s));
  EpiParams eg{};
  eg.vec = h->fw[7];
  eg.bias = h->fw[8];
  eg.out = h->at(h->off.pa_g);
  TRYS(gemm(h, F, Mmax, 4 * r, h->fw[6], 4 * r, M, r, 4 * r, EPI_PA_GATE, eg, s));
  const float* mparts[1] = {Mm};
  const int mw[1] = {r};
  void* Mb = h->at(h->off.pa_mb);
  TRY(concat_rows(mparts, mw, 1, M, Mb, h->act_bf16(), s));
  EpiParams eu{};
  eu.base = cv.h;
  eu.ldb = d;
  eu.gate = h->at(h->off.pa_g);
  eu.rowscale = cv.sH;
  eu.out = x;
  eu.ldo = d;
  return gemm(h, Mb, Mmax, r, h->fw[9], r, M, d, r, EPI_PA_UP, eu, s);
}

// D on x, then the output head and the per-row (conf, tok).  With
// masked_per_seq > 0 (and no logits requested) only the rows that still hold
// MASK go through the head: the sampler reads nothing else (carry-over), so
// the result is the same; they are gathered by the final RMSNorm and their
// (conf, tok) scattered back, the other rows get conf = -inf.
// With masked_per_seq > 0 the head runs only on the rows that hold MASK
// (masked_per_seq list entries per sequence, in h->off.idx); logits, if
// written, then follow the list order when compact_logits is set.
tadm_status run_D_head(tadm_handle* h, int B, int R, float* logits, cudaStream_t s, const int32_t* z = nullptr,
                       int ldz = 0, int masked_per_seq = 0, bool compact_logits = false) {
  const tadm_config& c = h->cfg;
  const int M = B * R, d = c.d_model;
  const int64_t Mmax = static_cast<int64_t>(h->max_batch) * h->max_rows;
  float* x = h->at<float>(h->off.x);
  TRYS(stack_fwd(h, c.n_shared + c.n_anchor, c.n_denoise, x, B, R, h->ctx, 0, s));
  void* norm = h->at(h->off.norm);
  const bool compact = masked_per_seq > 0 && z && (!logits || compact_logits);
  const int Mh = compact ? B * masked_per_seq : M;
  const int32_t* idx = compact ? h->at<int32_t>(h->off.idx) : nullptr;
  if (compact)
    TRY(masked_rows(z, ldz, B, R, c.vocab - 1, masked_per_seq, h->at<int32_t>(h->off.idx),
                    h->at<float>(h->off.conf), s));
  TRY(rmsnorm_rows(x, Mh, d, h->final_norm, c.dtype, c.norm_eps, norm, d, h->act_bf16(), s, idx));
  EpiParams e{};
  e.part = h->at<float>(h->off.part);
  e.mask_id = c.vocab - 1;
  e.logits = logits;
  e.ld_logits = c.vocab;
  TRYS(gemm(h, norm, Mmax, d, h->lm_head, d, Mh, c.vocab, d, EPI_LMHEAD, e, s));
  TRY(combine_partials(h->at<float>(h->off.part), Mh, h->n_part_tiles, h->at<float>(h->off.conf),
                       h->at<int32_t>(h->off.tok), s, idx));
  return TADM_OK;
}

// Causal fresh pass S -> A -> Phi(c, A(c)) -> D over rows appended to the context.
tadm_status fresh_pass(tadm_handle* h, const int32_t* z, int ldz, int B, int R, cudaStream_t s) {
  const tadm_config& c = h->cfg;
  if (h->max_ctx <= 0) return fail(h, TADM_ERR_STATE, "handle was created without KV context (max_ctx = 0)");
  if (h->ctx + R > h->max_ctx) return fail(h, TADM_ERR_STATE, "context full: %d + %d > %d", h->ctx, R, h->max_ctx);
  TRYS(run_S(h, z, ldz, B, R, 1, s));
  void* cache = h->at(h->off.h_int);
  TRYS(run_A(h, B, R, 1, cache, s));
  if (c.fusion == 1) {
    // fresh anchor: C = C0 gives M = 0, so H~ = H0 exactly (App. C.1)
    if (cudaMemcpyAsync(h->at(h->off.x), cache_view(c, cache, B, R).h, static_cast<size_t>(B) * R * c.d_model * 4,
                        cudaMemcpyDeviceToDevice, s) != cudaSuccess)
      return fail(h, TADM_ERR_CUDA, "copy H0 -> x failed");
  } else {
    TRYS(run_fusion(h, B, R, cache, s));
  }
  TRYS(stack_fwd(h, c.n_shared + c.n_anchor, c.n_denoise, h->at<float>(h->off.x), B, R, h->ctx, 1, s));
  h->ctx += R;
  h->counters.commit_passes += 1;
  return TADM_OK;
}

tadm_status check_ready(tadm_handle* h, int B, int R) {
  if (!h) return TADM_ERR_INVALID_ARG;
  if (!h->ws) return fail(h, TADM_ERR_STATE, "no workspace bound");
  if (B <= 0 || B > h->max_batch) return fail(h, TADM_ERR_INVALID_ARG, "batch %d outside 1..%d", B, h->max_batch);
  if (R <= 0 || R > h->max_rows) return fail(h, TADM_ERR_INVALID_ARG, "rows %d outside 1..%d", R, h->max_rows);
  if (h->batch && B != h->batch) return fail(h, TADM_ERR_STATE, "batch %d differs from the reset batch %d", B, h->batch);
  if (h->max_ctx > 0 && h->ctx + R > h->max_ctx)
    return fail(h, TADM_ERR_STATE, "rows beyond the KV capacity: %d + %d > %d", h->ctx, R, h->max_ctx);
  return TADM_OK;
}

// One reverse step after the (optional) refresh: c is already in the workspace.
tadm_status step_after_S(tadm_handle* h, int32_t* z, int ldz, int B, int R, int k, const void* cache,
                         const tadm_step_outputs* out, cudaStream_t s, int masked_per_seq = 0) {
  const tadm_config& c = h->cfg;
  TRYS(run_fusion(h, B, R, cache, s));
  const int M = B * R;
  if (out && out->fused &&
      cudaMemcpyAsync(out->fused, h->at(h->off.x), static_cast<size_t>(M) * c.d_model * 4, cudaMemcpyDeviceToDevice,
                      s) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "copy fused latent failed");
  TRYS(run_D_head(h, B, R, out ? out->logits : nullptr, s, z, ldz, masked_per_seq));
  float* conf = h->at<float>(h->off.conf);
  int32_t* tok = h->at<int32_t>(h->off.tok);
  if (out && out->conf && cudaMemcpyAsync(out->conf, conf, M * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "copy conf failed");
  if (out && out->tok && cudaMemcpyAsync(out->tok, tok, M * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "copy tok failed");
  TRY(topk_unmask(z, ldz, conf, tok, B, R, k, c.vocab - 1, out ? out->selected : nullptr, s));
  h->counters.shared_layers += c.n_shared;
  h->counters.denoise_layers += c.n_denoise;
  h->counters.denoise_steps += 1;
  return TADM_OK;
}

int unmask_count(int n, int T, int G) {
  return static_cast<int>((static_cast<int64_t>(n + 1) * G) / T - (static_cast<int64_t>(n) * G) / T);
}

std::vector<tadm_plan_event> make_plan(int P, int G, int T, int K, int bl) {
  std::vector<tadm_plan_event> ev;
  const int nblocks = bl > 0 ? G / bl : 1;
  const int Gb = bl > 0 ? bl : G;
  if (bl > 0) ev.push_back({0, -1, 0, 0});
  for (int b = 0; b < nblocks; ++b) {
    for (int n = 0; n < T; ++n) {
      if (n % K == 0) ev.push_back({1, b, n, 0});
      ev.push_back({2, b, n, unmask_count(n, T, Gb)});
    }
    if (bl > 0) ev.push_back({3, b, 0, 0});
  }
  (void)P;
  return ev;
}

const char* plan_args_error(int P, int G, int T, int K, int bl) {
  if (P < 0 || G <= 0) return "prompt_len >= 0 and gen_len > 0 required";
  if (T <= 0 || K <= 0) return "steps_per_block and K must be positive";
  if (bl < 0) return "block_len must be >= 0";
  if (bl > 0 && G % bl) return "gen_len must be a multiple of block_len";
  return nullptr;
}

}  // namespace

// =========================================================================== C ABI
// ReMDM schedule (the readings stated in tadm.h): {alpha_t, alpha_s, sigma, p_unmask} of step n.
double remdm_alpha(double t, int kind, double t_on, double t_off, double alpha_on) {
  if (kind == 0) return 1.0 - t;
  if (t > t_on) return alpha_on * (1.0 - t) / (1.0 - t_on);
  if (t >= t_off) return alpha_on;
  return alpha_on + (1.0 - alpha_on) * (t_off - t) / t_off;
}
void remdm_step_constants(int kind, int T, int n, double eta, double t_on, double t_off, double alpha_on,
                          double out[4]) {
  const double t = static_cast<double>(T - n) / T, s = static_cast<double>(T - n - 1) / T;
  const double a_t = remdm_alpha(t, kind, t_on, t_off, alpha_on), a_s = remdm_alpha(s, kind, t_on, t_off, alpha_on);
  double sigma_max = 1.0;
  if (a_t > 0.0) sigma_max = std::min(1.0, (1.0 - a_s) / a_t);
  const bool remask = kind == 0 || (t <= t_on && s >= t_off);
  const double sigma = remask ? std::min(eta, sigma_max) : 0.0;
  out[0] = a_t;
  out[1] = a_s;
  out[2] = sigma;
  out[3] = (a_s - (1.0 - sigma) * a_t) / (1.0 - a_t);
}
const char* remdm_args_error(int kind, double eta, double t_on, double t_off, double alpha_on) {
  if (kind != 0 && kind != 1) return "kind must be 0 (Cap) or 1 (Loop)";
  if (!(eta >= 0.0)) return "eta must be >= 0";
  if (kind == 1 && !(0.0 < t_off && t_off < t_on && t_on < 1.0 && 0.0 < alpha_on && alpha_on < 1.0))
    return "Loop needs 0 < t_off < t_on < 1 and 0 < alpha_on < 1";
  return nullptr;
}

extern "C" {

const char* tadm_status_string(tadm_status s) {
  switch (s) {
    case TADM_OK: return "ok";
    case TADM_ERR_INVALID_ARG: return "invalid argument";
    case TADM_ERR_UNSUPPORTED: return "unsupported";
    case TADM_ERR_CUDA: return "CUDA error";
    case TADM_ERR_OOM: return "workspace too small";
    case TADM_ERR_TIMEOUT: return "kernel wait timed out";
    case TADM_ERR_STATE: return "invalid state";
  }
  return "unknown status";
}

int tadm_weight_count(const tadm_config* cfg) {
  if (!valid_config(cfg, nullptr)) return -1;
  return static_cast<int>(inventory(cfg).names.size());
}

tadm_status tadm_weight_info(const tadm_config* cfg, int index, char* name, int name_cap, int64_t* rows,
                             int64_t* cols) {
  if (!valid_config(cfg, nullptr)) return TADM_ERR_INVALID_ARG;
  Inventory inv = inventory(cfg);
  if (index < 0 || index >= static_cast<int>(inv.names.size())) return TADM_ERR_INVALID_ARG;
  if (name && name_cap > 0) {
    std::snprintf(name, static_cast<size_t>(name_cap), "%s", inv.names[index].c_str());
  }
  if (rows) *rows = inv.rows[index];
  if (cols) *cols = inv.cols[index];
  return TADM_OK;
}

tadm_status tadm_create(const tadm_config* cfg, const void* const* weights, int n_weights, int max_batch,
                        int max_rows, int max_ctx, tadm_handle** out) {
  if (!out) return TADM_ERR_INVALID_ARG;
  *out = nullptr;
  std::string why;
  if (!valid_config(cfg, &why)) return TADM_ERR_INVALID_ARG;
  if (max_batch <= 0 || max_rows <= 0 || max_ctx < 0) return TADM_ERR_INVALID_ARG;
  const tadm_config& c = *cfg;
  // shapes the kernels of this build run
  if (c.dtype == 1) {
    if (c.head_dim != 64 && c.head_dim != 128) return TADM_ERR_UNSUPPORTED;
    if (c.d_model % 64 || c.ffn % 128) return TADM_ERR_UNSUPPORTED;
    if (c.fusion == 1 && (c.fusion_rank > 256 || (c.fusion_rank / c.fusion_heads != 64 &&
                                                  c.fusion_rank / c.fusion_heads != 128)))
      return TADM_ERR_UNSUPPORTED;
  } else {
    if (64 % c.head_dim || (c.head_dim != 32 && c.head_dim != 64)) return TADM_ERR_UNSUPPORTED;
    if (c.d_model % 32 || c.ffn % 32) return TADM_ERR_UNSUPPORTED;
    if (c.fusion == 1 && (c.fusion_rank > 64 || (c.fusion_rank / c.fusion_heads != 32 &&
                                                 c.fusion_rank / c.fusion_heads != 64)))
      return TADM_ERR_UNSUPPORTED;
  }
  Inventory inv = inventory(cfg);
  if (!weights || n_weights != static_cast<int>(inv.names.size())) return TADM_ERR_INVALID_ARG;
  for (int i = 0; i < n_weights; ++i)
    if (!weights[i] || (reinterpret_cast<uintptr_t>(weights[i]) & 15)) return TADM_ERR_INVALID_ARG;
  tadm_handle* h = new (std::nothrow) tadm_handle();
  if (!h) return TADM_ERR_OOM;
  h->cfg = c;
  h->inv = inv;
  h->w.assign(weights, weights + n_weights);
  h->max_batch = max_batch;
  h->max_rows = max_rows;
  h->max_ctx = max_ctx;
  h->L_total = c.n_shared + c.n_anchor + c.n_denoise;
  int i = 0;
  h->embed = weights[i++];
  for (int l = 0; l < h->L_total; ++l) {
    LayerW L{};
    L.attn_norm = weights[i++];
    L.wqkv = weights[i++];
    if (c.qk_norm) {
      L.q_norm = weights[i++];
      L.k_norm = weights[i++];
    }
    L.wo = weights[i++];
    if (c.sandwich_norm) L.post_attn = weights[i++];
    L.ffn_norm = weights[i++];
    L.wgu = weights[i++];
    L.wdown = weights[i++];
    if (c.sandwich_norm) L.post_ffn = weights[i++];
    // layer l of the whole backbone is global iff global_every == 0 or (l + 1) % global_every == 0
    L.global = c.global_every == 0 || (l + 1) % c.global_every == 0;
    L.window = L.global ? 0 : c.sliding_window;
    h->layers.push_back(L);
  }
  // fusion tensors (10 for fusion 0 and 1, none for fusion 2), in inventory order
  const int n_fusion = static_cast<int>(inv.names.size()) - i - (c.tied_lm_head ? 1 : 2);
  if (n_fusion < 0 || n_fusion > static_cast<int>(sizeof(h->fw) / sizeof(h->fw[0]))) {
    delete h;
    return TADM_ERR_INVALID_ARG;
  }
  for (int f = 0; f < n_fusion; ++f) h->fw[f] = weights[i++];
  h->final_norm = weights[i++];
  h->lm_head = c.tied_lm_head ? h->embed : weights[i++];
  if (i != static_cast<int>(inv.names.size())) {
    delete h;
    return TADM_ERR_INVALID_ARG;
  }
  layout(h);
  *out = h;
  return TADM_OK;
}

void tadm_destroy(tadm_handle* h) {
  if (h) {
    tadm_probe_enable(h, 0);
    if (h->gexec) cudaGraphExecDestroy(h->gexec);
    if (h->gev_in) cudaEventDestroy(h->gev_in);
    if (h->gev_out) cudaEventDestroy(h->gev_out);
    if (h->gstream) cudaStreamDestroy(h->gstream);
  }
  delete h;
}

tadm_status tadm_probe_enable(tadm_handle* h, int max_launches) {
  if (!h || max_launches < 0) return TADM_ERR_INVALID_ARG;
  for (cudaEvent_t e : h->probe_ev) cudaEventDestroy(e);
  h->probe_ev.clear();
  h->probe_flops.clear();
  h->probe_bytes.clear();
  h->probe_next = 0;
  if (max_launches == 0) return TADM_OK;
  h->probe_ev.resize(2 * static_cast<size_t>(max_launches));
  for (auto& e : h->probe_ev)
    if (cudaEventCreate(&e) != cudaSuccess) return fail(h, TADM_ERR_CUDA, "cudaEventCreate failed");
  h->probe_flops.assign(max_launches, 0.0);
  h->probe_bytes.assign(max_launches, 0.0);
  h->probe_kind.assign(max_launches, 0);
  return TADM_OK;
}

tadm_status tadm_probe_breakdown(tadm_handle* h, int n_kinds, int64_t* launches, double* ms, double* flops,
                                 double* bytes) {
  if (!h || n_kinds <= 0 || !launches || !ms || !flops) return TADM_ERR_INVALID_ARG;
  for (int k = 0; k < n_kinds; ++k) {
    launches[k] = 0;
    ms[k] = flops[k] = 0.0;
    if (bytes) bytes[k] = 0.0;
  }
  if (h->probe_next > 0 && cudaEventSynchronize(h->probe_ev[2 * h->probe_next - 1]) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "probe event sync failed");
  for (int i = 0; i < h->probe_next; ++i) {
    const int k = h->probe_kind[i];
    if (k < 0 || k >= n_kinds) continue;
    float t = 0.0f;
    if (cudaEventElapsedTime(&t, h->probe_ev[2 * i], h->probe_ev[2 * i + 1]) != cudaSuccess)
      return fail(h, TADM_ERR_CUDA, "probe elapsed time failed");
    launches[k] += 1;
    ms[k] += t;
    flops[k] += h->probe_flops[i];
    if (bytes) bytes[k] += h->probe_bytes[i];
  }
  return TADM_OK;
}

tadm_status tadm_probe_read(tadm_handle* h, int64_t* launches, double* total_ms, double* total_flops) {
  if (!h) return TADM_ERR_INVALID_ARG;
  double ms = 0.0, fl = 0.0;
  if (h->probe_next > 0 && cudaEventSynchronize(h->probe_ev[2 * h->probe_next - 1]) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "probe event sync failed");
  int64_t n_gemm = 0;
  for (int i = 0; i < h->probe_next; ++i) {
    if (h->probe_kind[i] >= kProbeAttention) continue;   // GEMM launches only
    float t = 0.0f;
    if (cudaEventElapsedTime(&t, h->probe_ev[2 * i], h->probe_ev[2 * i + 1]) != cudaSuccess)
      return fail(h, TADM_ERR_CUDA, "probe elapsed time failed");
    ms += t;
    fl += h->probe_flops[i];
    ++n_gemm;
  }
  if (launches) *launches = n_gemm;
  if (total_ms) *total_ms = ms;
  if (total_flops) *total_flops = fl;
  h->probe_next = 0;
  return TADM_OK;
}

const char* tadm_last_error(const tadm_handle* h) { return h ? h->err.c_str() : "NULL handle"; }

tadm_status tadm_workspace_size(const tadm_handle* h, size_t* bytes) {
  if (!h || !bytes) return TADM_ERR_INVALID_ARG;
  *bytes = h->ws_need;
  return TADM_OK;
}

tadm_status tadm_bind_workspace(tadm_handle* h, void* dev_ptr, size_t bytes) {
  if (!h || !dev_ptr) return TADM_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(dev_ptr) & 255) return fail(h, TADM_ERR_INVALID_ARG, "workspace not 256-byte aligned");
  if (bytes < h->ws_need) return fail(h, TADM_ERR_OOM, "workspace %zu < %zu bytes", bytes, h->ws_need);
  // a graph captured on the previous workspace must never replay on the new one
  if (h->gexec) {
    cudaGraphExecDestroy(h->gexec);
    h->gexec = nullptr;
  }
  std::memset(h->gkey, 0, sizeof(h->gkey));
  std::memset(h->gkey_seen, 0, sizeof(h->gkey_seen));
  h->ws = static_cast<char*>(dev_ptr);
  h->ws_bytes = bytes;
  const int n_pos = h->kv_stride + h->max_rows;
  cudaStream_t s = nullptr;
  TRY(rope_table(h->at<float2>(h->off.rope), n_pos, h->cfg.head_dim, h->cfg.rope_theta, s));
  if (h->off.rope_g != h->off.rope)
    TRY(rope_table(h->at<float2>(h->off.rope_g), n_pos, h->cfg.head_dim, h->cfg.rope_theta_global, s));
  if (cudaMemsetAsync(h->status(), 0, 256, s) != cudaSuccess) return fail(h, TADM_ERR_CUDA, "memset failed");
  // K / V positions that were never written are read with zero weight; keep them finite
  if (cudaMemsetAsync(h->at(h->off.kv), 0, h->off.attn - h->off.kv, s) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "memset failed");
  if (cudaStreamSynchronize(s) != cudaSuccess) return fail(h, TADM_ERR_CUDA, "bind: %s", cudaGetErrorString(cudaGetLastError()));
  return TADM_OK;
}

tadm_status tadm_cache_size(const tadm_handle* h, int batch, int rows, size_t* bytes) {
  if (!h || !bytes || batch <= 0 || rows <= 0) return TADM_ERR_INVALID_ARG;
  *bytes = cache_bytes(h->cfg, batch, rows);
  return TADM_OK;
}

tadm_status tadm_reset(tadm_handle* h, int batch) {
  if (!h) return TADM_ERR_INVALID_ARG;
  if (batch <= 0 || batch > h->max_batch) return fail(h, TADM_ERR_INVALID_ARG, "batch %d outside 1..%d", batch, h->max_batch);
  h->batch = batch;
  h->ctx = 0;
  h->counters = tadm_counters{};
  if (h->ws && cudaMemsetAsync(h->status(), 0, 256, nullptr) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "memset failed");
  return TADM_OK;
}

tadm_status tadm_prefill(tadm_handle* h, const int32_t* prompt, int batch, int prompt_len, tadm_stream stream) {
  TRYS(check_ready(h, batch, prompt_len));
  if (!prompt) return fail(h, TADM_ERR_INVALID_ARG, "prompt is NULL");
  h->last_stream = stream;
  return fresh_pass(h, prompt, prompt_len, batch, prompt_len, stream);
}

tadm_status tadm_commit_block(tadm_handle* h, const int32_t* x_block, int batch, int rows, tadm_stream stream) {
  TRYS(check_ready(h, batch, rows));
  if (!x_block) return fail(h, TADM_ERR_INVALID_ARG, "x_block is NULL");
  h->last_stream = stream;
  return fresh_pass(h, x_block, rows, batch, rows, stream);
}

tadm_status tadm_anchor_forward(tadm_handle* h, const int32_t* x_t, int batch, int rows, int t, void* h_cache,
                                tadm_stream stream) {
  (void)t;
  TRYS(check_ready(h, batch, rows));
  if (!x_t || !h_cache) return fail(h, TADM_ERR_INVALID_ARG, "NULL pointer");
  h->last_stream = stream;
  TRYS(run_S(h, x_t, rows, batch, rows, 0, stream));
  TRYS(run_A(h, batch, rows, 0, h_cache, stream));
  h->counters.anchor_layers += h->cfg.n_anchor;
  h->counters.anchor_calls += 1;
  return TADM_OK;
}

tadm_status tadm_denoise_step(tadm_handle* h, int32_t* x_t, int batch, int rows, int t, int T, int n_masked_at_start,
                              const void* h_cache, const tadm_step_outputs* out, tadm_stream stream) {
  TRYS(check_ready(h, batch, rows));
  if (!x_t || !h_cache) return fail(h, TADM_ERR_INVALID_ARG, "NULL pointer");
  if (T <= 0 || t < 1 || t > T || n_masked_at_start < 0 || n_masked_at_start > rows)
    return fail(h, TADM_ERR_INVALID_ARG, "need 1 <= t <= T and 0 <= n_masked_at_start <= rows");
  h->last_stream = stream;
  const int k = unmask_count(T - t, T, n_masked_at_start);
  TRYS(run_S(h, x_t, rows, batch, rows, 0, stream));
  return step_after_S(h, x_t, rows, batch, rows, k, h_cache, out, stream);
}

tadm_status tadm_plan(int prompt_len, int gen_len, int steps_per_block, int K, int block_len, tadm_plan_event* events,
                      int cap, int* n_events) {
  if (plan_args_error(prompt_len, gen_len, steps_per_block, K, block_len)) return TADM_ERR_INVALID_ARG;
  std::vector<tadm_plan_event> ev = make_plan(prompt_len, gen_len, steps_per_block, K, block_len);
  if (n_events) *n_events = static_cast<int>(ev.size());
  for (int i = 0; i < cap && i < static_cast<int>(ev.size()); ++i) events[i] = ev[i];
  return TADM_OK;
}

tadm_status tadm_layer_cost(int L_S, int L_A, int L_D, int T, int K, int64_t* c_full, int64_t* c_cache) {
  if (L_S < 0 || L_A < 0 || L_D < 0 || T <= 0 || K <= 0) return TADM_ERR_INVALID_ARG;
  if (c_full) *c_full = static_cast<int64_t>(T) * (L_S + L_A + L_D);
  if (c_cache) *c_cache = static_cast<int64_t>(T) * (L_S + L_D) + static_cast<int64_t>((T + K - 1) / K) * L_A;
  return TADM_OK;
}

tadm_status generate_loop(tadm_handle* h, const int32_t* prompt, int batch, int prompt_len, int32_t* out,
                          int gen_len, int steps_per_block, int K, int block_len, cudaStream_t s);

tadm_status tadm_generate(tadm_handle* h, const int32_t* prompt, int batch, int prompt_len, int32_t* out, int gen_len,
                          int steps_per_block, int K, int block_len, tadm_stream stream) {
  if (!h) return TADM_ERR_INVALID_ARG;
  if (const char* e = plan_args_error(prompt_len, gen_len, steps_per_block, K, block_len))
    return fail(h, TADM_ERR_INVALID_ARG, "%s", e);
  if (!prompt || !out) return fail(h, TADM_ERR_INVALID_ARG, "NULL pointer");
  const int total = prompt_len + gen_len;
  const int R = block_len > 0 ? block_len : total;
  if (block_len > 0 && prompt_len == 0) return fail(h, TADM_ERR_INVALID_ARG, "block mode needs a prompt");
  if (block_len > 0 && (prompt_len > h->max_rows || total > h->max_ctx))
    return fail(h, TADM_ERR_INVALID_ARG, "block mode needs prompt_len <= max_rows and prompt+gen <= max_ctx");
  TRYS(tadm_reset(h, batch));
  TRYS(check_ready(h, batch, R));
  h->last_stream = stream;
  static const bool graphs_on = [] {
    const char* e = getenv("TADM_GRAPH");
    return !(e && e[0] == '0');
  }();
  const int64_t key[9] = {batch, prompt_len, gen_len, steps_per_block, K, block_len,
                          static_cast<int64_t>(reinterpret_cast<uintptr_t>(prompt)),
                          static_cast<int64_t>(reinterpret_cast<uintptr_t>(out)),
                          static_cast<int64_t>(reinterpret_cast<uintptr_t>(h->ws))};
  if (!graphs_on || !h->probe_flops.empty()) return generate_loop(h, prompt, batch, prompt_len, out, gen_len,
                                                                  steps_per_block, K, block_len, stream);
  const bool seen = std::memcmp(key, h->gkey_seen, sizeof(key)) == 0;
  std::memcpy(h->gkey_seen, key, sizeof(key));
  if (!seen && !(h->gexec && std::memcmp(key, h->gkey, sizeof(key)) == 0))   // first call: eager
    return generate_loop(h, prompt, batch, prompt_len, out, gen_len, steps_per_block, K, block_len, stream);
  if (!h->gstream) {
    if (cudaStreamCreateWithFlags(&h->gstream, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&h->gev_in, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&h->gev_out, cudaEventDisableTiming) != cudaSuccess)
      return fail(h, TADM_ERR_CUDA, "graph stream / events");
  }
  if (!(h->gexec && std::memcmp(key, h->gkey, sizeof(key)) == 0)) {
    // second identical call: capture the whole generation on the internal stream
    if (h->gexec) {
      cudaGraphExecDestroy(h->gexec);
      h->gexec = nullptr;
    }
    if (cudaStreamBeginCapture(h->gstream, cudaStreamCaptureModeThreadLocal) != cudaSuccess)
      return fail(h, TADM_ERR_CUDA, "begin graph capture");
    const tadm_status st = generate_loop(h, prompt, batch, prompt_len, out, gen_len, steps_per_block, K, block_len,
                                         h->gstream);
    cudaGraph_t g = nullptr;
    const cudaError_t ce = cudaStreamEndCapture(h->gstream, &g);
    if (st != TADM_OK) {
      if (g) cudaGraphDestroy(g);
      return st;
    }
    if (ce != cudaSuccess || !g) return fail(h, TADM_ERR_CUDA, "end graph capture: %s", cudaGetErrorString(ce));
    const cudaError_t ie = cudaGraphInstantiate(&h->gexec, g, 0);
    cudaGraphDestroy(g);
    if (ie != cudaSuccess) {
      h->gexec = nullptr;
      return fail(h, TADM_ERR_CUDA, "graph instantiate: %s", cudaGetErrorString(ie));
    }
    std::memcpy(h->gkey, key, sizeof(key));
    h->gcounters = h->counters;
    h->gctx = h->ctx;
  }
  // replay, ordered after the caller's stream and before its next work
  h->counters = h->gcounters;
  h->ctx = h->gctx;
  h->counters.kernel_launches = h->gcounters.kernel_launches;
  if (cudaEventRecord(h->gev_in, stream) != cudaSuccess || cudaStreamWaitEvent(h->gstream, h->gev_in, 0) != cudaSuccess ||
      cudaGraphLaunch(h->gexec, h->gstream) != cudaSuccess || cudaEventRecord(h->gev_out, h->gstream) != cudaSuccess ||
      cudaStreamWaitEvent(stream, h->gev_out, 0) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "graph launch");
  return TADM_OK;
}

// The issue loop of tadm_generate (Alg. 1 per block, prefill and commits).
tadm_status generate_loop(tadm_handle* h, const int32_t* prompt, int batch, int prompt_len, int32_t* out,
                          int gen_len, int steps_per_block, int K, int block_len, cudaStream_t s) {
  const int total = prompt_len + gen_len;
  const int R = block_len > 0 ? block_len : total;
  const tadm_config& c = h->cfg;
  TRY(fill_canvas(out, total, prompt, batch, prompt_len, total, c.vocab - 1, s));
  void* cache = h->at(h->off.h_int);
  bool have_c = false;  // a refresh computed c = S(z) for the step that follows it
  for (const tadm_plan_event& e : make_plan(prompt_len, gen_len, steps_per_block, K, block_len)) {
    int32_t* z = out + (block_len > 0 ? prompt_len + e.block * block_len : 0);
    switch (e.kind) {
      case 0:  // encoder prefill of the prompt
        TRYS(fresh_pass(h, out, total, batch, prompt_len, s));
        break;
      case 1:  // anchor refresh: h_cache <- A(S(z))
        TRYS(run_S(h, z, total, batch, R, 0, s));
        TRYS(run_A(h, batch, R, 0, cache, s));
        h->counters.anchor_layers += c.n_anchor;
        h->counters.anchor_calls += 1;
        have_c = true;
        break;
      case 2: {  // denoising step with the (possibly stale) cache, then the sampler
        if (!have_c) TRYS(run_S(h, z, total, batch, R, 0, s));
        have_c = false;
        // positions of the active rows still masked before step n: G_b - floor(n G_b / T)
        const int Gb = block_len > 0 ? block_len : gen_len;
        const int masked = Gb - static_cast<int>(static_cast<int64_t>(e.n) * Gb / steps_per_block);
        TRYS(step_after_S(h, z, total, batch, R, e.k, cache, nullptr, s, masked));
        break;
      }
      case 3:  // commit the finished block into the KV context
        TRYS(fresh_pass(h, z, total, batch, block_len, s));
        break;
    }
  }
  return TADM_OK;
}

tadm_status tadm_sync_status(tadm_handle* h) {
  if (!h) return TADM_ERR_INVALID_ARG;
  if (!h->ws) return fail(h, TADM_ERR_STATE, "no workspace bound");
  if (cudaStreamSynchronize(h->last_stream) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "%s", cudaGetErrorString(cudaGetLastError()));
  int st = 0;
  if (cudaMemcpy(&st, h->status(), sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return fail(h, TADM_ERR_CUDA, "status read failed");
  if (st & kErrTimeout) return fail(h, TADM_ERR_TIMEOUT, "a kernel gave up a bounded wait (status 0x%x)", st);
  if (st & kErrLayout) return fail(h, TADM_ERR_CUDA, "a kernel found its shared memory misaligned (status 0x%x)", st);
  return TADM_OK;
}

tadm_status tadm_get_counters(const tadm_handle* h, tadm_counters* out) {
  if (!h || !out) return TADM_ERR_INVALID_ARG;
  *out = h->counters;
  return TADM_OK;
}

// --------------------------------------------------------------- building blocks
tadm_status tadm_gemm(const void* A, const void* B, void* C, int M, int N, int K, int lda, int ldb, int ldc, int dtype,
                      int c_dtype, tadm_stream stream) {
  if (!A || !B || !C || M < 0 || N < 0 || K < 0 || lda < K || ldb < K || ldc < N) return TADM_ERR_INVALID_ARG;
  if ((dtype != 0 && dtype != 1) || (c_dtype != 0 && c_dtype != 1)) return TADM_ERR_INVALID_ARG;
  GemmCall g{};
  g.A = A;
  g.B = B;
  g.M = M;
  g.N = N;
  g.K = K;
  g.lda = lda;
  g.ldb = ldb;
  g.epi = EPI_STORE;
  g.ep.out = C;
  g.ep.ldo = ldc;
  g.ep.out_bf16 = c_dtype;
  const char* e = dtype ? gemm_tc(g, stream) : gemm_simt(g, stream);
  return e ? TADM_ERR_CUDA : TADM_OK;
}

tadm_status tadm_confidence(const float* logits, int rows, int vocab, int mask_id, float* conf, int32_t* tok,
                            tadm_stream stream) {
  if (!logits || !conf || !tok || rows < 0 || vocab < 2 || mask_id < 0 || mask_id >= vocab) return TADM_ERR_INVALID_ARG;
  return confidence_rows(logits, rows, vocab, vocab, mask_id, conf, tok, stream) ? TADM_ERR_CUDA : TADM_OK;
}

tadm_status tadm_topk_unmask(int32_t* z, int ldz, const float* conf, const int32_t* tok, int batch, int rows, int k,
                             int mask_id, int32_t* selected, tadm_stream stream) {
  if (!z || !conf || !tok || batch < 0 || rows < 0 || k < 0 || ldz < rows) return TADM_ERR_INVALID_ARG;
  return topk_unmask(z, ldz, conf, tok, batch, rows, k, mask_id, selected, stream) ? TADM_ERR_CUDA : TADM_OK;
}

tadm_status tadm_head_scratch_size(int rows, int vocab, int dtype, size_t* bytes) {
  if (!bytes || rows < 0 || vocab < 2 || (dtype != 0 && dtype != 1)) return TADM_ERR_INVALID_ARG;
  const int tiles = dtype ? gemm_tc_tiles_n(vocab, EPI_LMHEAD) : gemm_simt_tiles_n(vocab, EPI_LMHEAD);
  *bytes = static_cast<size_t>(rows) * tiles * 3 * sizeof(float);
  return TADM_OK;
}

tadm_status tadm_head_confidence(const void* x, const void* w, int rows, int d, int vocab, int mask_id, int dtype,
                                 void* scratch, size_t scratch_bytes, float* conf, int32_t* tok, tadm_stream stream) {
  size_t need = 0;
  if (tadm_head_scratch_size(rows, vocab, dtype, &need) != TADM_OK) return TADM_ERR_INVALID_ARG;
  if (!x || !w || !conf || !tok || d <= 0 || mask_id < 0 || mask_id >= vocab) return TADM_ERR_INVALID_ARG;
  if (rows == 0) return TADM_OK;
  if (!scratch || scratch_bytes < need) return TADM_ERR_INVALID_ARG;
  GemmCall g{};
  g.A = x;
  g.B = w;
  g.M = rows;
  g.N = vocab;
  g.K = d;
  g.lda = d;
  g.ldb = d;
  g.epi = EPI_LMHEAD;
  g.ep.part = static_cast<float*>(scratch);
  g.ep.mask_id = mask_id;
  const char* e = dtype ? gemm_tc(g, stream) : gemm_simt(g, stream);
  if (e) return TADM_ERR_CUDA;
  const int tiles = dtype ? gemm_tc_tiles_n(vocab, EPI_LMHEAD) : gemm_simt_tiles_n(vocab, EPI_LMHEAD);
  return combine_partials(static_cast<const float*>(scratch), rows, tiles, conf, tok, stream) ? TADM_ERR_CUDA
                                                                                               : TADM_OK;
}

tadm_status tadm_attention(const void* q, const void* k, const void* v, void* o, int batch, int n_heads, int n_kv_heads,
                           int head_dim, int rows, int ctx, int kv_stride, int causal, int window, int dtype,
                           tadm_stream stream) {
  if (!q || !k || !v || !o || batch < 0 || n_heads <= 0 || n_kv_heads <= 0 || rows < 0 || ctx < 0 || window < 0)
    return TADM_ERR_INVALID_ARG;
  AttnCall a{q, k, v, o, batch, n_heads, n_kv_heads, head_dim, rows, ctx, kv_stride, causal, dtype, nullptr};
  a.window = window;
  return attention(a, stream) ? TADM_ERR_CUDA : TADM_OK;
}

tadm_status tadm_remdm_schedule(int kind, int T, int n, double eta, double t_on, double t_off, double alpha_on,
                                double out[4]) {
  if (!out || T < 1 || n < 0 || n >= T || remdm_args_error(kind, eta, t_on, t_off, alpha_on))
    return TADM_ERR_INVALID_ARG;
  remdm_step_constants(kind, T, n, eta, t_on, t_off, alpha_on, out);
  return TADM_OK;
}

tadm_status tadm_remdm_uniforms(uint64_t seed, int step, int batch, int rows, float* out, tadm_stream stream) {
  if (!out || batch <= 0 || rows <= 0 || step < 0) return TADM_ERR_INVALID_ARG;
  return remdm_uniforms(seed, step, batch, rows, out, stream) ? TADM_ERR_CUDA : TADM_OK;
}

tadm_status tadm_remdm_update(int32_t* z, int ldz, const float* logits, int ld_logits, int batch, int rows,
                              int first_gen, int vocab, int mask_id, double sigma, double p_unmask, float top_p,
                              uint64_t seed, int step, int32_t* action, tadm_stream stream) {
  if (!z || !logits || !action || batch <= 0 || rows <= 0 || ldz < rows || vocab < 2 || ld_logits < vocab ||
      mask_id < 0 || mask_id >= vocab || first_gen < 0 || step < 0 || !(top_p > 0.0f && top_p <= 1.0f) ||
      !(sigma >= 0.0 && sigma <= 1.0) || !(p_unmask >= 0.0 && p_unmask <= 1.0 + 1e-12))
    return TADM_ERR_INVALID_ARG;
  if (remdm_decide(z, ldz, batch, rows, first_gen, mask_id, sigma, p_unmask, seed, step, action, stream) ||
      remdm_sample(logits, ld_logits, batch * rows, nullptr, action, z, ldz, batch, rows, vocab, mask_id, top_p, seed,
                   step, stream))
    return TADM_ERR_CUDA;
  return TADM_OK;
}

tadm_status tadm_generate_remdm(tadm_handle* h, const int32_t* prompt, int batch, int prompt_len, int32_t* out,
                                int gen_len, int steps, int K, int kind, double eta, float top_p, uint64_t seed,
                                float* logits_scratch, size_t scratch_bytes, tadm_stream stream) {
  if (!h) return TADM_ERR_INVALID_ARG;
  constexpr double t_on = 0.55, t_off = 0.05, alpha_on = 0.9;
  if (const char* e = remdm_args_error(kind, eta, t_on, t_off, alpha_on)) return fail(h, TADM_ERR_INVALID_ARG, "%s", e);
  if (!prompt || !out || !logits_scratch) return fail(h, TADM_ERR_INVALID_ARG, "NULL pointer");
  if (prompt_len < 0 || gen_len <= 0 || steps < 1 || K < 1 || !(top_p > 0.0f && top_p <= 1.0f))
    return fail(h, TADM_ERR_INVALID_ARG, "need gen_len > 0, steps >= 1, K >= 1, 0 < top_p <= 1");
  if (h->max_ctx > 0) return fail(h, TADM_ERR_INVALID_ARG, "the ReMDM sampler runs single-block canvases (max_ctx = 0)");
  const tadm_config& c = h->cfg;
  const int total = prompt_len + gen_len, R = total;
  const size_t need = static_cast<size_t>(batch) * gen_len * c.vocab * sizeof(float);
  if (scratch_bytes < need) return fail(h, TADM_ERR_INVALID_ARG, "logits_scratch needs %zu bytes", need);
  TRYS(tadm_reset(h, batch));
  TRYS(check_ready(h, batch, R));
  h->last_stream = stream;
  cudaStream_t s = stream;
  const int mask = c.vocab - 1;
  int32_t* act = h->at<int32_t>(h->off.act);
  int32_t* idx = h->at<int32_t>(h->off.idx);
  int* cnt = h->at<int>(h->off.cnt);
  const int bound = batch * gen_len;           // unmasking rows of a step: at most every generated position
  const int64_t Mmax = static_cast<int64_t>(h->max_batch) * h->max_rows;
  TRY(fill_canvas(out, total, prompt, batch, prompt_len, total, mask, s));
  void* cache = h->at(h->off.h_int);
  for (int n = 0; n < steps; ++n) {
    TRYS(run_S(h, out, total, batch, R, 0, s));
    if (n % K == 0) {                          // Alg. 1 refresh test (T - i) mod K = 0
      TRYS(run_A(h, batch, R, 0, cache, s));
      h->counters.anchor_layers += c.n_anchor;
      h->counters.anchor_calls += 1;
    }
    TRYS(run_fusion(h, batch, R, cache, s));
    float* x = h->at<float>(h->off.x);
    TRYS(stack_fwd(h, c.n_shared + c.n_anchor, c.n_denoise, x, batch, R, 0, 0, s));
    // the decisions need only the draws and z_t: decide (remasks applied), then
    // run the output head on the unmasking rows alone (device count)
    double k[4];
    remdm_step_constants(kind, steps, n, eta, t_on, t_off, alpha_on, k);
    TRY(remdm_decide(out, total, batch, R, prompt_len, mask, k[2], k[3], seed, n, act, s));
    TRY(remdm_rows(act, batch * R, bound, idx, cnt, s));
    void* norm = h->at(h->off.norm);
    TRY(rmsnorm_rows(x, bound, c.d_model, h->final_norm, c.dtype, c.norm_eps, norm, c.d_model, h->act_bf16(), s, idx));
    EpiParams e{};
    e.part = h->at<float>(h->off.part);
    e.mask_id = mask;
    e.logits = logits_scratch;
    e.ld_logits = c.vocab;
    TRYS(gemm(h, norm, Mmax, c.d_model, h->lm_head, c.d_model, bound, c.vocab, c.d_model, EPI_LMHEAD, e, s, false, cnt));
    TRY(remdm_sample(logits_scratch, c.vocab, bound, idx, act, out, total, batch, R, c.vocab, mask, top_p, seed, n, s,
                     cnt));
    h->counters.shared_layers += c.n_shared;
    h->counters.denoise_layers += c.n_denoise;
    h->counters.denoise_steps += 1;
  }
  return TADM_OK;
}

}  // extern "C"

// ------------------------------------------------------------ entropy-bound sampler
namespace {

// Caller scratch of the entropy-bound generation, in this order (each
// segment 256-byte aligned): logits fp32 [n, V]; with self-conditioning
// q = exp((l - max) / tau) [n, V] and E^T [d, V] (model element type), the
// unnormalised signal q E fp32 [n, d] and Z = sum q fp32 [n]; H fp32 [n];
// n = batch * gen_len.
struct EbScratch {
  size_t logits, p, et, sig, zs, ent, total;
};

EbScratch eb_layout(const tadm_config& c, int batch, int gen_len, int self_cond) {
  const size_t n = static_cast<size_t>(batch) * gen_len, es = c.dtype ? 2 : 4;
  EbScratch L{};
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o = align_up(o + bytes, 256);
    return at;
  };
  L.logits = take(n * c.vocab * 4);
  if (self_cond) {
    L.p = take(n * c.vocab * es);
    L.et = take(static_cast<size_t>(c.d_model) * c.vocab * es);
    L.sig = take(n * c.d_model * 4);
    L.zs = take(n * 4);
  }
  L.ent = take(n * 4);
  L.total = o;
  return L;
}

const char* eb_args_error(int steps, int K, double eta, double tau_max, double tau_min, int self_cond) {
  if (steps < 1 || K < 1) return "need steps >= 1 and K >= 1";
  if (eta != eta) return "eta is NaN";
  if (!(tau_min > 0.0) || !(tau_max >= tau_min) || !(tau_max < 1e30)) return "need 0 < tau_min <= tau_max";
  if (self_cond != 0 && self_cond != 1) return "self_cond must be 0 or 1";
  return nullptr;
}

}  // namespace

extern "C" {

tadm_status tadm_eb_update(int32_t* z, int ldz, const float* logits, int ld_logits, int batch, int rows, int first_gen,
                           int vocab, int mask_id, double tau, double eta, int last, uint64_t seed, int step,
                           float* entropy, void* probs, int probs_dtype, int ld_probs, float* z_sum,
                           tadm_stream stream) {
  const int G = rows - first_gen;
  if (!z || !logits || batch <= 0 || rows <= 0 || first_gen < 0 || G <= 0 || ldz < rows || vocab < 2 ||
      ld_logits < vocab || mask_id < 0 || mask_id >= vocab || step < 0 || !(tau > 0.0) || eta != eta ||
      (last != 0 && last != 1) || (!last && !entropy) || (probs && ld_probs < vocab) ||
      (probs_dtype != 0 && probs_dtype != 1) || G > eb_max_gen())
    return TADM_ERR_INVALID_ARG;
  cudaStream_t s = stream;
  if (eb_row(logits, ld_logits, batch, rows, first_gen, z, ldz, vocab, mask_id, static_cast<float>(1.0 / tau), last,
             seed, step, nullptr, 0, last ? nullptr : probs, probs_dtype, ld_probs, entropy, z_sum, s))
    return TADM_ERR_CUDA;
  if (!last && eb_accept(entropy, batch, rows, first_gen, z, ldz, vocab, eta, seed, step, s)) return TADM_ERR_CUDA;
  return TADM_OK;
}

tadm_status tadm_eb_scratch_bytes(const tadm_handle* h, int batch, int gen_len, int self_cond, size_t* bytes) {
  if (!h || !bytes || batch <= 0 || gen_len <= 0 || (self_cond != 0 && self_cond != 1)) return TADM_ERR_INVALID_ARG;
  *bytes = eb_layout(h->cfg, batch, gen_len, self_cond).total;
  return TADM_OK;
}

tadm_status tadm_generate_entropy_bound(tadm_handle* h, const int32_t* prompt, int batch, int prompt_len,
                                        int32_t* out, int gen_len, int steps, int K, double eta, double tau_max,
                                        double tau_min, int self_cond, uint64_t seed, void* scratch,
                                        size_t scratch_bytes, tadm_stream stream) {
  if (!h) return TADM_ERR_INVALID_ARG;
  if (const char* e = eb_args_error(steps, K, eta, tau_max, tau_min, self_cond))
    return fail(h, TADM_ERR_INVALID_ARG, "%s", e);
  if (!prompt || !out || !scratch) return fail(h, TADM_ERR_INVALID_ARG, "NULL pointer");
  if (prompt_len < 0 || gen_len <= 0 || gen_len > eb_max_gen())
    return fail(h, TADM_ERR_INVALID_ARG, "need 0 < gen_len <= %d", eb_max_gen());
  if (h->max_ctx > 0)
    return fail(h, TADM_ERR_INVALID_ARG, "the entropy-bound sampler runs single-block canvases (max_ctx = 0)");
  const tadm_config& c = h->cfg;
  if (self_cond && c.dtype && c.vocab % 8)
    return fail(h, TADM_ERR_INVALID_ARG, "self-conditioning on a bf16 model needs vocab % 8 == 0");
  const EbScratch L = eb_layout(c, batch, gen_len, self_cond);
  if (scratch_bytes < L.total || reinterpret_cast<uintptr_t>(scratch) % 256)
    return fail(h, TADM_ERR_INVALID_ARG, "scratch needs %zu bytes, 256-byte aligned", L.total);
  const int total = prompt_len + gen_len, R = total, n_rows = batch * gen_len;
  TRYS(tadm_reset(h, batch));
  TRYS(check_ready(h, batch, R));
  h->last_stream = stream;
  cudaStream_t s = stream;
  const int mask = c.vocab - 1;
  char* base = static_cast<char*>(scratch);
  float* logits = reinterpret_cast<float*>(base + L.logits);
  float* ent = reinterpret_cast<float*>(base + L.ent);
  void* p = self_cond ? base + L.p : nullptr;
  void* et = self_cond ? base + L.et : nullptr;
  float* sig = self_cond ? reinterpret_cast<float*>(base + L.sig) : nullptr;
  float* zs = self_cond ? reinterpret_cast<float*>(base + L.zs) : nullptr;
  const int head_tiles = c.dtype ? gemm_tc_tiles_n(c.vocab, EPI_LMHEAD) : gemm_simt_tiles_n(c.vocab, EPI_LMHEAD);
  int32_t* idx = h->at<int32_t>(h->off.idx);
  const int64_t Mmax = static_cast<int64_t>(h->max_batch) * h->max_rows;
  if (self_cond) TRY(transpose(h->embed, c.vocab, c.d_model, c.dtype, et, s));   // E^T [d, V] for s = p E
  TRY(fill_canvas(out, total, prompt, batch, prompt_len, total, mask, s));
  TRY(eb_noise(out, total, batch, R, prompt_len, c.vocab, seed, steps, s));       // z_T: noise of step T
  TRY(eb_rows(idx, batch, R, prompt_len, s));
  void* cache = h->at(h->off.h_int);
  for (int i = 0; i < steps; ++i) {
    const int n = steps - i;                      // Alg. 2's n = T .. 1
    TRYS(run_S(h, out, total, batch, R, 0, s, self_cond && i > 0 ? sig : nullptr, prompt_len, zs));
    if (i % K == 0) {                             // Alg. 1 refresh test (T - i) mod K = 0
      TRYS(run_A(h, batch, R, 0, cache, s));
      h->counters.anchor_layers += c.n_anchor;
      h->counters.anchor_calls += 1;
    }
    TRYS(run_fusion(h, batch, R, cache, s));
    float* x = h->at<float>(h->off.x);
    TRYS(stack_fwd(h, c.n_shared + c.n_anchor, c.n_denoise, x, batch, R, 0, 0, s));
    void* norm = h->at(h->off.norm);
    TRY(rmsnorm_rows(x, n_rows, c.d_model, h->final_norm, c.dtype, c.norm_eps, norm, c.d_model, h->act_bf16(), s,
                     idx));
    EpiParams e{};
    e.part = h->at<float>(h->off.part);
    e.mask_id = mask;
    e.logits = logits;
    e.ld_logits = c.vocab;
    TRYS(gemm(h, norm, Mmax, c.d_model, h->lm_head, c.d_model, n_rows, c.vocab, c.d_model, EPI_LMHEAD, e, s));
    const double tau = tau_min + (tau_max - tau_min) * n / steps;
    const int last = n == 1;
    // max and argmax from the head's partials; q = exp((l - max) / tau) and Z for s = (q E) / Z
    TRY(eb_row(logits, c.vocab, batch, R, prompt_len, out, total, c.vocab, mask, static_cast<float>(1.0 / tau), last,
               seed, i, e.part, head_tiles, last ? nullptr : p, c.dtype, c.vocab, ent, zs, s));
    if (!last) {
      if (self_cond) {                            // q E; the next step's embedding adds it divided by Z
        EpiParams es{};
        es.out = sig;
        es.ldo = c.d_model;
        TRYS(gemm(h, p, n_rows, c.vocab, et, c.vocab, n_rows, c.d_model, c.vocab, EPI_STORE, es, s, true));
      }
      TRY(eb_accept(ent, batch, R, prompt_len, out, total, c.vocab, eta, seed, i, s));
    }
    h->counters.shared_layers += c.n_shared;
    h->counters.denoise_layers += c.n_denoise;
    h->counters.denoise_steps += 1;
  }
  return TADM_OK;
}

}  // extern "C"
