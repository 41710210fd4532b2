// C-ABI of libflashbon.so: model set-up, the host dispatcher of the draft path and the
// single-op entry points. See include/flashbon.h for the contract of each call.
//
// The dispatcher turns (schedule, skip_mask, proxy_plan) into one launch list per step:
// a computed block is its chain of kernels (norms, tcgen05 GEMMs, attention), a run of
// proxied blocks (skipped blocks between them are no-ops, Eq. 6) is ONE proxy_add
// launch, a skipped block launches nothing. Cached contributions Delta_l are written by
// the epilogue of the block's last GEMM into a ring of anchor slots; slots are assigned
// on the host from the plan, so only contributions some later proxy reads are stored.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <atomic>
#include <mutex>
#include <thread>
#include <string>
#include <vector>

#include "../../include/flashbon.h"
#include "kernels.h"

bool fb_pdl_enabled() {
  static const bool on = getenv("FB_NO_PDL") == nullptr;
  return on;
}
namespace {
thread_local bool g_prev_op_is_kernel = false;
}
bool fb_prev_op_is_kernel() { return g_prev_op_is_kernel; }
void fb_set_prev_op_is_kernel(bool v) { g_prev_op_is_kernel = v; }

namespace {

thread_local std::string g_last_error;

fb_status fail(fb_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

#define CK(call)                                                                    \
  do {                                                                              \
    cudaError_t e_ = (call);                                                        \
    if (e_ != cudaSuccess)                                                          \
      return fail(FB_ECUDA, "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_), \
                  __FILE__, __LINE__);                                              \
  } while (0)
#define CKS(call)                  \
  do {                             \
    fb_status s_ = (call);         \
    if (s_ != FB_OK) return s_;    \
  } while (0)

enum WKind { W_MAT, W_VEC };
struct WEntry {
  std::string name;
  size_t numel;
  WKind kind;
};

std::vector<WEntry> weight_table(const fb_cfg& c) {
  const size_t D = c.dim, F = c.ffn, PD = (size_t)c.latent_c * c.patch * c.patch;
  std::vector<WEntry> t = {
      {"patch.w", D * PD, W_MAT}, {"patch.b", D, W_VEC},
      {"time.w1", D * c.freq_dim, W_MAT}, {"time.b1", D, W_VEC},
      {"time.w2", D * D, W_MAT}, {"time.b2", D, W_VEC},
      {"mod.w", 6 * D * D, W_MAT}, {"mod.b", 6 * D, W_VEC},
      {"text.w1", D * c.text_dim, W_MAT}, {"text.b1", D, W_VEC},
      {"text.w2", D * D, W_MAT}, {"text.b2", D, W_VEC},
      {"head.table", 2 * D, W_VEC}, {"head.w", PD * D, W_MAT}, {"head.b", PD, W_VEC},
  };
  for (int l = 0; l < c.depth; ++l) {
    const std::string p = "blocks." + std::to_string(l) + ".";
    std::vector<WEntry> b = {
        {p + "table", 6 * D, W_VEC},
        {p + "attn.wqkv", 3 * D * D, W_MAT}, {p + "attn.bqkv", 3 * D, W_VEC},
        {p + "attn.norm_q", D, W_VEC}, {p + "attn.norm_k", D, W_VEC},
        {p + "attn.wo", D * D, W_MAT}, {p + "attn.bo", D, W_VEC},
        {p + "norm3.w", D, W_VEC}, {p + "norm3.b", D, W_VEC},
        {p + "cross.wq", D * D, W_MAT}, {p + "cross.bq", D, W_VEC},
        {p + "cross.wkv", 2 * D * D, W_MAT}, {p + "cross.bkv", 2 * D, W_VEC},
        {p + "cross.norm_q", D, W_VEC}, {p + "cross.norm_k", D, W_VEC},
        {p + "cross.wo", D * D, W_MAT}, {p + "cross.bo", D, W_VEC},
        {p + "ffn.w1", F * D, W_MAT}, {p + "ffn.b1", F, W_VEC},
        {p + "ffn.w2", D * F, W_MAT}, {p + "ffn.b2", D, W_VEC},
    };
    t.insert(t.end(), b.begin(), b.end());
  }
  return t;
}

bool ln_width_ok(int D) {
  switch (D) {
    case 128: case 256: case 512: case 1024: case 1536: case 2048: case 3072: case 4096:
    case 5120:
      return true;
  }
  return false;
}

fb_status check_cfg(const fb_cfg* c) {
  if (!c) return fail(FB_EINVAL, "cfg is NULL");
  if (c->depth < 1 || c->dim < 1 || c->heads < 1 || c->ffn < 1 || c->text_len < 1 ||
      c->text_dim < 1 || c->latent_c < 1 || c->patch < 1 || c->max_n < 1 || c->freq_dim < 2)
    return fail(FB_EINVAL, "cfg: sizes must be positive");
  if (c->head_dim != 64 && c->head_dim != 128)
    return fail(FB_EINVAL, "cfg: head_dim must be 64 or 128");
  if (c->heads * c->head_dim != c->dim) return fail(FB_EINVAL, "cfg: dim != heads * head_dim");
  if (!ln_width_ok(c->dim)) return fail(FB_EINVAL, "cfg: unsupported dim %d", c->dim);
  if (c->latent_h % c->patch || c->latent_w % c->patch || c->latent_h < c->patch ||
      c->latent_w < c->patch)
    return fail(FB_EINVAL, "cfg: latent size must be a positive multiple of patch");
  const int pd = c->latent_c * c->patch * c->patch;
  if (pd % 8 || pd > 64 || 256 % pd) return fail(FB_EINVAL, "cfg: C*p*p must be 8, 16, 32 or 64");
  if (c->ffn % 8 || c->text_dim % 8 || c->freq_dim % 16)
    return fail(FB_EINVAL, "cfg: ffn, text_dim multiple of 8; freq_dim multiple of 16");
  if (!(c->eps_ln > 0) || !(c->eps_rms > 0) || !(c->rope_theta > 1))
    return fail(FB_EINVAL, "cfg: eps must be > 0 and rope_theta > 1");
  return FB_OK;
}

struct Layer {
  bf16 *wqkv, *wo, *cq, *ckv, *co, *w1, *w2;
  float *table, *bqkv, *nq, *nk, *bo, *n3w, *n3b, *cbq, *cbkv, *cnq, *cnk, *cbo, *b1, *b2;
};

struct Pending {
  int kind;
  cudaEvent_t a, b;
};

}  // namespace

struct fb_model {
  fb_cfg c;
  int dev = 0;  // the device current at fb_init_model; every launch of the model runs there
  int P, PD, gh, gw;
  size_t Mmax;
  int num_sms;      // SMs the model's launches may use (fb_set_sm_budget), <= dev_sms
  int dev_sms = 0;  // the device's SMs
  cudaStream_t own = nullptr, st = nullptr;
  // weights
  void* wmat = nullptr;  // bf16 matrices
  void* wvec = nullptr;  // fp32 vectors (tables contiguous: per-layer tables first)
  bf16 *patch_w, *time_w1, *time_w2, *mod_w, *text_w1, *text_w2, *head_w;
  float *patch_b, *time_b1, *time_b2, *mod_b, *text_b1, *text_b2, *head_table, *head_b;
  float* tables;  // [depth][6][D]
  std::vector<Layer> L;
  // tensor-core patch embedding and head (C p p % 64 == 0, D % 128 == 0): bf16 patch rows
  // [Mmax][PD]; head weights and bias zero-padded to npad = PD rounded up to 128 rows, and
  // the head output [Mmax][npad] fp32. Null: the CUDA-core kernels.
  bf16* patch_a = nullptr;
  bf16* head_wp = nullptr;
  float* head_bp = nullptr;
  float* vbuf = nullptr;
  int npad = 0;
  // activations
  float *hA = nullptr, *hB = nullptr;
  bf16 *act = nullptr, *qkv = nullptr, *ao = nullptr, *cqb = nullptr, *ffh = nullptr;
  float* ctx_f = nullptr;
  bf16 *ctx_b = nullptr, *ctx_h = nullptr, *ctx_p = nullptr, *kvctx = nullptr;
  bf16* kvctx_u = nullptr;  // unconditional context (guidance), allocated on first use
  float* noise = nullptr;   // device copy of host SDE draws, grown on demand
  size_t noise_elems = 0;
  bool text_ready = false;
  float *emb = nullptr, *th1 = nullptr, *temb = nullptr, *mod = nullptr, *modl = nullptr,
        *hmod = nullptr;
  float2* rope = nullptr;
  float* zbuf = nullptr;
  bf16* anchors = nullptr;
  size_t anchor_elems = 0;
  int* derr = nullptr;
  int* herr = nullptr;  // pinned
  // cached draft state (fb_draft_ex with keep_state): per layer the anchor slot of its
  // last computed contribution (-1: none) and that step's t; rows of nr candidates per slot
  bool state_valid = false;
  int state_n = 0, state_nr = 0;
  std::vector<int> state_slot;
  std::vector<float> state_tau;
  // offloads in flight: a copy stream, and per anchor slot the event of the last copy
  // reading it (pending until a later write has waited for it)
  cudaStream_t copy_st = nullptr;
  std::vector<cudaEvent_t> slot_ev;
  std::vector<char> slot_pending;
  size_t pending_elems = 0;  // slot size (elements) the pending copies were issued with
  // stream-K workspace of the 2-SM GEMM: partial accumulators and per-tile counters
  // (zero between launches; reset after a device error)
  float* sk_ws = nullptr;
  int* sk_ctr = nullptr;
  int sk_clusters = 0;
  // statistics
  unsigned timing_mask = 0;
  int op_repeat = 1;
  fb_kstat stats[FB_K_COUNT];
  std::vector<Pending> pending;
  std::vector<cudaEvent_t> ev_pool;
  std::vector<void*> allocs;
};

namespace {

// ---- allocation helpers -------------------------------------------------------------
// Host-side failure injection (fb_test_fail_alloc): device allocations are counted from
// the last arming, and the one whose index equals g_fail_at fails as cudaMalloc would.
std::atomic<long> g_alloc_calls{0};
std::atomic<long> g_fail_at{-1};

fb_status dalloc(fb_model* m, void** p, size_t bytes) {
  *p = nullptr;
  if (bytes == 0) bytes = 16;
  if (g_alloc_calls.fetch_add(1) == g_fail_at.load())
    return fail(FB_ENOMEM, "cudaMalloc(%zu bytes) failed: injected failure", bytes);
  cudaError_t e = cudaMalloc(p, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(FB_ENOMEM, "cudaMalloc(%zu bytes) failed: %s", bytes, cudaGetErrorString(e));
  }
  m->allocs.push_back(*p);
  return FB_OK;
}
template <typename T>
fb_status dalloc_t(fb_model* m, T** p, size_t n) {
  return dalloc(m, reinterpret_cast<void**>(p), n * sizeof(T));
}

// ---- statistics ---------------------------------------------------------------------
struct KTimer {
  fb_model* m;
  int kind;
  cudaEvent_t a = nullptr, b = nullptr;
  KTimer(fb_model* mm, int k, double flops, double bytes, int nlaunch = 1) : m(mm), kind(k) {
    m->stats[k].launches += nlaunch;
    m->stats[k].flops += flops;
    m->stats[k].bytes += bytes;
    if (m->timing_mask & (1u << k)) {
      a = get();
      b = get();
      if (a && b) {
        cudaEventRecord(a, m->st);
        fb_stream_op_not_kernel();
      }
    }
  }
  cudaEvent_t get() {
    if (!m->ev_pool.empty()) {
      cudaEvent_t e = m->ev_pool.back();
      m->ev_pool.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    return e;
  }
  ~KTimer() {
    if (a && b) {
      cudaEventRecord(b, m->st);
      fb_stream_op_not_kernel();
      m->pending.push_back({kind, a, b});
    } else {
      if (a) m->ev_pool.push_back(a);
      if (b) m->ev_pool.push_back(b);
    }
  }
};

void collect_timings(fb_model* m) {
  for (auto& p : m->pending) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, p.a, p.b) == cudaSuccess) m->stats[p.kind].ms += ms;
    else cudaGetLastError();
    m->ev_pool.push_back(p.a);
    m->ev_pool.push_back(p.b);
  }
  m->pending.clear();
}

// Starts an API call: clears the device error word. Work the caller queued on the
// stream before the call is not one of our kernels either.
fb_status begin_call(fb_model* m) {
  fb_stream_op_not_kernel();
  CK(cudaMemsetAsync(m->derr, 0, sizeof(int), m->st));
  return FB_OK;
}
// Ends an API call: waits for the stream, checks the device error word.
fb_status end_call(fb_model* m) {
  fb_stream_op_not_kernel();
  CK(cudaMemcpyAsync(m->herr, m->derr, sizeof(int), cudaMemcpyDeviceToHost, m->st));
  CK(cudaStreamSynchronize(m->st));
  collect_timings(m);
  if (*m->herr != 0 && m->sk_ctr) {
    // a kernel that gave up may have left stream-K counters counted in
    fb_stream_op_not_kernel();
    CK(cudaMemsetAsync(m->sk_ctr, 0, (size_t)m->sk_clusters * SK_CTR_PER_CLUSTER * sizeof(int),
                       m->st));
    CK(cudaStreamSynchronize(m->st));
  }
  if (*m->herr == FB_DEVERR_WAIT_TIMEOUT)
    return fail(FB_ECUDA, "device wait timed out (a kernel gave up after its time limit)");
  if (*m->herr != 0) return fail(FB_ECUDA, "device error %d", *m->herr);
  return FB_OK;
}

// ---- kernel wrappers with statistics ------------------------------------------------
// impl: 0 automatic, 1 CUDA-core kernel, 2 the 1-SM tcgen05 kernel, 3 the 2-SM kernel
// over whole tiles, 4 the 2-SM kernel with the stream-K split
fb_status run_gemm(fb_model* m, const GemmArgs& g0, int impl = 0) {
  GemmArgs g = g0;
  g.sk_ws = m->sk_ws;
  g.sk_ctr = m->sk_ctr;
  g.sk_clusters = m->sk_clusters;
  g.sk_mode = impl == 3 ? 1 : impl == 4 ? 2 : 0;
  const double flops = 2.0 * g.M * (double)g.N * g.K;
  double bytes = 2.0 * ((double)g.M * g.K + (double)g.N * g.K);
  bytes += (g.kind <= EPI_GELU_BF16) ? 2.0 * g.M * g.N : 8.0 * g.M * g.N;
  if (g.kind == EPI_RESID_DELTA) bytes += 6.0 * g.M * g.N;
  if (impl != 1 && gemm_tc_supported(g)) {
    KTimer t(m, FB_K_GEMM_TC, flops, bytes);
    CK(gemm_tc(g, m->derr, m->num_sms, m->st, impl == 2));
  } else {
    KTimer t(m, FB_K_GEMM_SIMT, flops, bytes);
    CK(gemm_simt(g, m->st));
  }
  return FB_OK;
}

GemmArgs gemm_args(int M, int N, int K, const bf16* A, const bf16* W, const float* bias,
                   int kind, void* out) {
  GemmArgs g{};
  g.M = M; g.N = N; g.K = K;
  g.A = A; g.lda = K;
  g.W = W; g.ldw = K;
  g.kind = kind;
  g.epi.bias = bias;
  g.epi.out = out;
  g.epi.ldo = N;
  return g;
}

// impl: 0 automatic (tcgen05 for head_dim 128), 1 the mma.sync kernel, 2 / 3 the tcgen05
// kernel with 128- / 256-query CTAs
fb_status run_attn(fb_model* m, const AttnArgs& a0, int kind, int impl = 0) {
  AttnArgs a = a0;
  a.tc_variant = impl >= 2 ? impl - 1 : 0;
  a.sms = m->num_sms;
  const double flops = 4.0 * a.batch * a.heads * (double)a.Lq * a.Lkv * a.head_dim;
  const double kvb = (a.kv_batch_rows ? a.batch : 1) * 2.0 * a.Lkv * a.heads * a.head_dim * 2;
  const double bytes = 2.0 * a.batch * a.Lq * (double)a.heads * a.head_dim * 2 + kvb;
  KTimer t(m, kind, flops, bytes);
  if (impl != 1 && attention_tc_supported(a)) CK(attention_tc(a, m->derr, m->st));
  else if (impl >= 2) return fail(FB_EINVAL, "the tcgen05 attention kernel needs head_dim 128");
  else CK(attention(a, m->st));
  return FB_OK;
}

fb_status run_ln(fb_model* m, const float* x, bf16* out, int rows, float mb, const float* mul,
                 const float* add) {
  KTimer t(m, FB_K_NORM, 8.0 * rows * m->c.dim, 6.0 * rows * m->c.dim);
  CK(ln_mod(x, out, rows, m->c.dim, m->c.eps_ln, mb, mul, add, m->st));
  return FB_OK;
}

fb_status run_qkn(fb_model* m, bf16* x, int rows, int ld, int nseg, int col0, const float* w0,
                  int col1, const float* w1, const float2* rope) {
  KTimer t(m, FB_K_QKNORM, 6.0 * rows * nseg * m->c.dim, 4.0 * rows * nseg * m->c.dim);
  CK(qk_norm_rope(x, rows, ld, m->c.dim, nseg, col0, w0, col1, w1, m->c.eps_rms, rope, m->P,
                  m->c.head_dim, m->st));
  return FB_OK;
}

// ---- text encoding (once per call) --------------------------------------------------
fb_status encode_text(fb_model* m, const float* ctx, bf16* kv_dst) {
  const fb_cfg& c = m->c;
  const size_t nctx = (size_t)c.text_len * c.text_dim;
  cudaPointerAttributes at{};
  const float* src = ctx;
  if (cudaPointerGetAttributes(&at, ctx) != cudaSuccess) cudaGetLastError();
  if (at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged) {
    CK(cudaMemcpyAsync(m->ctx_f, ctx, nctx * sizeof(float), cudaMemcpyHostToDevice, m->st));
    fb_stream_op_not_kernel();
    src = m->ctx_f;
  }
  {
    KTimer t(m, FB_K_SMALL, 0, 6.0 * nctx);
    CK(f32_to_bf16(src, m->ctx_b, nctx, m->st));
  }
  const int T = c.text_len, D = c.dim;
  CKS(run_gemm(m, gemm_args(T, D, c.text_dim, m->ctx_b, m->text_w1, m->text_b1, EPI_GELU_BF16,
                            m->ctx_h)));
  CKS(run_gemm(m, gemm_args(T, D, D, m->ctx_h, m->text_w2, m->text_b2, EPI_BF16, m->ctx_p)));
  for (int l = 0; l < c.depth; ++l) {
    bf16* kv = kv_dst + (size_t)l * T * 2 * D;
    CKS(run_gemm(m, gemm_args(T, 2 * D, D, m->ctx_p, m->L[l].ckv, m->L[l].cbkv, EPI_BF16, kv)));
    CKS(run_qkn(m, kv, T, 2 * D, 1, 0, m->L[l].cnk, 0, m->L[l].cnk, nullptr));
  }
  if (kv_dst == m->kvctx) m->text_ready = true;
  return FB_OK;
}

// ---- per-step conditioning: temb, mod, per-layer modulation, head modulation ---------
// have_emb: m->emb already holds the sinusoid of t (written by the previous step's
// Euler kernel)
fb_status time_embed(fb_model* m, float t, bool have_emb = false) {
  const fb_cfg& c = m->c;
  const int D = c.dim;
  KTimer k(m, FB_K_SMALL, 2.0 * D * (c.freq_dim + D + 6.0 * D),
           2.0 * D * (c.freq_dim + D + 6.0 * D), have_emb ? 4 : 5);
  if (!have_emb) CK(timestep_sincos(t, c.freq_dim, m->emb, m->st));
  CK(gemv(m->time_w1, m->time_b1, m->emb, m->th1, D, c.freq_dim, 0, 1, m->st));
  CK(gemv(m->time_w2, m->time_b2, m->th1, m->temb, D, D, 0, 0, m->st));
  CK(gemv(m->mod_w, m->mod_b, m->temb, m->mod, 6 * D, D, 1, 0, m->st));
  CK(mod_prepare(m->mod, m->tables, c.depth, D, m->modl, m->head_table, m->temb, m->hmod, m->st));
  return FB_OK;
}

// ---- one block B_l (Eq. 7) on h = hA (rows M), optional contribution write ----------
// n: candidates (rows n*P). n_uncond > 0: the last n_uncond candidates are the
// unconditional rows of guidance and attend to the unconditional text context.
fb_status block_forward(fb_model* m, int l, float* h, int n, bf16* delta, int n_uncond = 0) {
  const fb_cfg& c = m->c;
  const int D = c.dim, M = n * m->P;
  const Layer& w = m->L[l];
  const float* md = m->modl + (size_t)l * 6 * D;
  const float *s1 = md, *c1 = md + D, *g1 = md + 2 * D, *s2 = md + 3 * D, *c2 = md + 4 * D,
              *g2 = md + 5 * D;
  float* hB = m->hB;
  // self-attention branch
  CKS(run_ln(m, h, m->act, M, 1.f, c1, s1));
  CKS(run_gemm(m, gemm_args(M, 3 * D, D, m->act, w.wqkv, w.bqkv, EPI_BF16, m->qkv)));
  CKS(run_qkn(m, m->qkv, M, 3 * D, 2, 0, w.nq, D, w.nk, m->rope));
  {
    AttnArgs a{};
    a.Q = m->qkv; a.K = m->qkv + D; a.V = m->qkv + 2 * D; a.O = m->ao;
    a.ldq = a.ldk = a.ldv = 3 * D; a.ldo = D;
    a.batch = n; a.Lq = m->P; a.Lkv = m->P; a.kv_batch_rows = m->P;
    a.heads = c.heads; a.head_dim = c.head_dim;
    CKS(run_attn(m, a, FB_K_ATTN_SELF));
  }
  {
    GemmArgs g = gemm_args(M, D, D, m->ao, w.wo, w.bo, EPI_RESID, hB);
    g.epi.resid = h;
    g.epi.gate = g1;
    CKS(run_gemm(m, g));
  }
  // cross-attention branch
  CKS(run_ln(m, hB, m->act, M, 0.f, w.n3w, w.n3b));
  CKS(run_gemm(m, gemm_args(M, D, D, m->act, w.cq, w.cbq, EPI_BF16, m->cqb)));
  CKS(run_qkn(m, m->cqb, M, D, 1, 0, w.cnq, 0, w.cnq, nullptr));
  for (int part = 0; part < (n_uncond ? 2 : 1); ++part) {
    const int n0 = part ? n - n_uncond : 0, nb = n_uncond ? (part ? n_uncond : n - n_uncond) : n;
    const bf16* kv = (part ? m->kvctx_u : m->kvctx) + (size_t)l * c.text_len * 2 * D;
    AttnArgs a{};
    a.Q = m->cqb + (size_t)n0 * m->P * D; a.K = kv; a.V = kv + D;
    a.O = m->ao + (size_t)n0 * m->P * D;
    a.ldq = D; a.ldk = a.ldv = 2 * D; a.ldo = D;
    a.batch = nb; a.Lq = m->P; a.Lkv = c.text_len; a.kv_batch_rows = 0;
    a.heads = c.heads; a.head_dim = c.head_dim;
    CKS(run_attn(m, a, FB_K_ATTN_CROSS));
  }
  {
    GemmArgs g = gemm_args(M, D, D, m->ao, w.co, w.cbo, EPI_RESID, hB);
    g.epi.resid = hB;
    CKS(run_gemm(m, g));
  }
  // feed-forward branch; the last epilogue writes h and, if asked, Delta = h_new - h_old
  CKS(run_ln(m, hB, m->act, M, 1.f, c2, s2));
  CKS(run_gemm(m, gemm_args(M, c.ffn, D, m->act, w.w1, w.b1, EPI_GELU_BF16, m->ffh)));
  {
    GemmArgs g = gemm_args(M, D, c.ffn, m->ffh, w.w2, w.b2, delta ? EPI_RESID_DELTA : EPI_RESID, h);
    g.epi.resid = hB;
    g.epi.gate = g2;
    g.epi.base = h;
    g.epi.delta = delta;
    CKS(run_gemm(m, g));
  }
  return FB_OK;
}

// ---- plan analysis ------------------------------------------------------------------
struct Action {
  int type;   // 0 compute, 1 proxy run
  int layer;  // compute: layer
  int slot;   // compute: anchor slot for Delta, -1 = none
  std::vector<std::pair<int, double>> terms;  // proxy: (slot, coefficient)
};
struct Plan {
  std::vector<std::vector<Action>> steps;
  int n_slots = 0;
  // keep: per layer the slot holding its last computed contribution (-1: none) and t
  std::vector<int> keep_slot;
  std::vector<float> keep_tau;
  // warm start: per layer the slot its cached-state contribution is uploaded to (-1: none)
  std::vector<int> warm_src;
};

fb_status analyse_plan(const fb_cfg& c, const float* sched, int S, const uint8_t* skip,
                       const int32_t* proxy, Plan* out, bool keep = false) {
  const int L = c.depth;
  auto is_skip = [&](int k, int l) { return skip && skip[(size_t)k * L + l] != 0; };
  auto code = [&](int k, int l) { return proxy ? proxy[(size_t)k * L + l] : -1; };
  // computed steps per layer; anchors per proxy; last use per (step, layer)
  std::vector<std::vector<int>> computed(L);
  std::map<std::pair<int, int>, std::vector<int>> anchors;
  std::map<std::pair<int, int>, int> last_use;  // (step, layer) -> last proxy step using it
  for (int k = 0; k < S; ++k)
    for (int l = 0; l < L; ++l) {
      const int32_t cd = code(k, l);
      if (cd == -1) {
        if (!is_skip(k, l)) computed[l].push_back(k);
        continue;
      }
      if (is_skip(k, l)) return fail(FB_EPLAN, "step %d layer %d: skipped and proxied", k, l);
      if (cd < 0) return fail(FB_EPLAN, "step %d layer %d: bad proxy code %d", k, l, cd);
      const int src = cd & 0xFFFF, order = cd >> 16;
      if (order > 2) return fail(FB_EPLAN, "step %d layer %d: order %d > 2", k, l, order);
      if (src >= k) return fail(FB_EPLAN, "step %d layer %d: source step %d not earlier", k, l, src);
      const auto& cl = computed[l];
      if (std::find(cl.begin(), cl.end(), src) == cl.end())
        return fail(FB_EPLAN, "step %d layer %d: not computed at source step %d", k, l, src);
      std::vector<int> an;
      for (auto it = cl.rbegin(); it != cl.rend() && (int)an.size() < order + 1; ++it)
        if (*it <= src) an.push_back(*it);
      for (int s : an) last_use[{s, l}] = k;
      anchors[{k, l}] = an;
    }
  // the cached state: each layer's last computed contribution stays until the end
  if (keep)
    for (int l = 0; l < L; ++l)
      if (!computed[l].empty()) last_use[{computed[l].back(), l}] = S;
  // slot assignment: per layer a pool; a slot is free once its last user has run
  std::vector<std::vector<int>> free_at(L);  // per layer: for each slot, step after which it is free
  std::vector<int> slot_base(L, 0);
  std::map<std::pair<int, int>, int> slot_of;  // (step, layer) -> local slot
  for (int k = 0; k < S; ++k)
    for (int l = 0; l < L; ++l) {
      auto lu = last_use.find({k, l});
      if (lu == last_use.end()) continue;
      auto& pool = free_at[l];
      int s = -1;
      for (size_t i = 0; i < pool.size(); ++i)
        if (pool[i] < k) { s = (int)i; break; }
      if (s < 0) { s = (int)pool.size(); pool.push_back(0); }
      pool[s] = lu->second;
      slot_of[{k, l}] = s;
    }
  int total = 0;
  for (int l = 0; l < L; ++l) { slot_base[l] = total; total += (int)free_at[l].size(); }
  out->n_slots = total;
  out->keep_slot.assign(keep ? L : 0, -1);
  out->keep_tau.assign(keep ? L : 0, std::nanf(""));
  if (keep)
    for (int l = 0; l < L; ++l)
      if (!computed[l].empty()) {
        const int k = computed[l].back();
        out->keep_slot[l] = slot_base[l] + slot_of[{k, l}];
        out->keep_tau[l] = sched[k];
      }
  out->steps.assign(S, {});
  for (int k = 0; k < S; ++k) {
    auto& acts = out->steps[k];
    for (int l = 0; l < L; ++l) {
      if (is_skip(k, l)) continue;  // Eq. 6: identity, no launch
      const int32_t cd = code(k, l);
      if (cd == -1) {
        Action a{0, l, -1, {}};
        auto so = slot_of.find({k, l});
        if (so != slot_of.end()) a.slot = slot_base[l] + so->second;
        acts.push_back(a);
        continue;
      }
      // Eqs. 3-5 as weights of the anchors h1, h2, h3 (most recent first):
      // h~ = h1 + a (h1 - h2) + a^2/2 (h1 - 2 h2 + h3), a = (t - tau1) / (tau1 - tau2)
      const auto& an = anchors[{k, l}];
      const double t = sched[k];
      std::vector<double> w;
      if (an.size() == 1) {
        w = {1.0};
      } else {
        const double tau1 = sched[an[0]], tau2 = sched[an[1]];
        const double a = (t - tau1) / (tau1 - tau2);
        if (an.size() == 2) w = {1.0 + a, -a};
        else w = {1.0 + a + 0.5 * a * a, -a - a * a, 0.5 * a * a};
      }
      if (acts.empty() || acts.back().type != 1) acts.push_back(Action{1, -1, -1, {}});
      for (size_t i = 0; i < an.size(); ++i)
        acts.back().terms.push_back({slot_base[l] + slot_of[{an[i], l}], w[i]});
    }
  }
  return FB_OK;
}

// Refine plan warm-started from a cached state: at steps < warm every layer the state
// holds (held[l]) is an order-0 proxy of its own slot (slot_of[l], coefficient 1);
// everything else computes. Runs of consecutive proxied layers form one proxy action.
void warm_plan(int L, int S, int warm, const std::vector<int>& slot_of, Plan* out) {
  out->steps.assign(S, {});
  out->n_slots = 0;
  out->warm_src = slot_of;
  for (int l = 0; l < L; ++l)
    if (slot_of[l] >= 0) out->n_slots = std::max(out->n_slots, slot_of[l] + 1);
  for (int k = 0; k < S; ++k)
    for (int l = 0; l < L; ++l) {
      auto& acts = out->steps[k];
      if (k < warm && slot_of[l] >= 0) {
        if (acts.empty() || acts.back().type != 1) acts.push_back(Action{1, -1, -1, {}});
        acts.back().terms.push_back({slot_of[l], 1.0});
      } else {
        acts.push_back(Action{0, l, -1, {}});
      }
    }
}

fb_status check_schedule(const float* s, int n_steps) {
  if (!s) return fail(FB_EINVAL, "schedule is NULL");
  for (int i = 0; i <= n_steps; ++i)
    if (!(s[i] >= 0.f && s[i] <= 1.f)) return fail(FB_EINVAL, "schedule[%d] outside [0, 1]", i);
  for (int i = 0; i < n_steps; ++i)
    if (!(s[i + 1] < s[i])) return fail(FB_EINVAL, "schedule not strictly decreasing at %d", i);
  return FB_OK;
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

struct SampOpts {
  bool guided = false;
  float w = 1.f;
  float sde_a = 0.f;
  const float* noise = nullptr;  // device, [S][n][C][H][W]
};

// The sampler loop shared by fb_draft and fb_refine (latents z on the device). With
// guidance the batch holds 2n candidates' rows: n conditional, then n unconditional.
// Before a write into anchor slot `slot` of slot_elems elements: the compute stream waits
// for the offload copies still reading any part of it. Pending copies are tracked per
// slot of the geometry (pending_elems) they were issued with.
fb_status wait_slot(fb_model* m, int slot, size_t slot_elems) {
  if (slot < 0) return FB_OK;
  const size_t b = (size_t)slot * slot_elems, e = b + slot_elems;
  for (int s = 0; s < (int)m->slot_pending.size(); ++s) {
    const size_t sb = (size_t)s * m->pending_elems, se = sb + m->pending_elems;
    if (!m->slot_pending[s] || se <= b || e <= sb) continue;
    fb_stream_op_not_kernel();
    CK(cudaStreamWaitEvent(m->st, m->slot_ev[s], 0));
    m->slot_pending[s] = 0;
  }
  return FB_OK;
}

// The contribution cache holds at least `need` elements; growing it first lets every
// copy still reading it finish.
fb_status ensure_anchors(fb_model* m, size_t need) {
  if (need <= m->anchor_elems) return FB_OK;
  fb_stream_op_not_kernel();
  CK(cudaStreamSynchronize(m->st));
  if (m->copy_st) {
    CK(cudaStreamSynchronize(m->copy_st));
    std::fill(m->slot_pending.begin(), m->slot_pending.end(), 0);
  }
  m->state_valid = false;
  if (m->anchors) {
    cudaFree(m->anchors);
    m->allocs.erase(std::find(m->allocs.begin(), m->allocs.end(), (void*)m->anchors));
    m->anchors = nullptr;
    m->anchor_elems = 0;
  }
  CKS(dalloc_t(m, &m->anchors, need));
  m->anchor_elems = need;
  return FB_OK;
}

fb_status sample(fb_model* m, float* z, int n, const float* sched, int S, const Plan& plan,
                 const SampOpts& so) {
  const fb_cfg& c = m->c;
  const int nr = so.guided ? 2 * n : n;  // candidates' rows in the batch
  const size_t slot_elems = (size_t)nr * m->P * c.dim;
  const size_t need = slot_elems * plan.n_slots;
  CKS(ensure_anchors(m, need));
  const int M = nr * m->P;
  const size_t zn = (size_t)n * c.latent_c * c.latent_h * c.latent_w;
  // with the tensor-core head, each step's Euler kernel also writes the next step's
  // sinusoidal embedding and patch rows (step 0 computes its own)
  const bool fused_next = m->vbuf && m->patch_a;
  for (int k = 0; k < S; ++k) {
    const float t = sched[k], t1 = sched[k + 1];
    const bool from_prev = fused_next && k > 0;
    CKS(time_embed(m, t, from_prev));
    for (int u = 0; u < (so.guided ? 2 : 1); ++u) {
      float* hu = m->hA + (size_t)u * n * m->P * c.dim;
      const bool rows_ready = from_prev || u > 0;
      KTimer kt(m, FB_K_EMBED, 2.0 * n * m->P * (double)c.dim * m->PD,
                (rows_ready ? 2.0 : 4.0) * n * m->P * (double)(c.dim + m->PD),
                m->patch_a ? (rows_ready ? 1 : 2) : 1);
      if (m->patch_a) {
        // tensor cores: bf16 patch rows, then h = patches W_p^T + b_p (fp32, no residual)
        if (!rows_ready)
          CK(patchify(z, n, c.latent_c, c.latent_h, c.latent_w, c.patch, m->patch_a, m->st));
        const GemmArgs g = gemm_args(n * m->P, c.dim, m->PD, m->patch_a, m->patch_w, m->patch_b,
                                     EPI_RESID, hu);
        CK(gemm_tc(g, m->derr, m->num_sms, m->st));
      } else {
        CK(patch_embed(z, n, c.latent_c, c.latent_h, c.latent_w, c.patch, m->patch_w, m->patch_b,
                       c.dim, hu, m->st));
      }
    }
    for (const Action& a : plan.steps[k]) {
      if (a.type == 0) {
        bf16* d = a.slot >= 0 ? m->anchors + (size_t)a.slot * slot_elems : nullptr;
        CKS(wait_slot(m, a.slot, slot_elems));
        CKS(block_forward(m, a.layer, m->hA, nr, d, so.guided ? n : 0));
      } else {
        for (size_t i0 = 0; i0 < a.terms.size(); i0 += FB_PROXY_MAX_TERMS) {
          ProxyTerms pt{};
          pt.n = (int)std::min(a.terms.size() - i0, (size_t)FB_PROXY_MAX_TERMS);
          for (int i = 0; i < pt.n; ++i) {
            pt.ptr[i] = m->anchors + (size_t)a.terms[i0 + i].first * slot_elems;
            pt.coef[i] = (float)a.terms[i0 + i].second;
          }
          KTimer kt(m, FB_K_PROXY, 2.0 * pt.n * (double)M * c.dim,
                    (double)M * c.dim * (8.0 + 2.0 * pt.n));
          CK(proxy_add(m->hA, (size_t)M * c.dim, pt, m->st));
        }
      }
    }
    CKS(run_ln(m, m->hA, m->act, M, 1.f, m->hmod + c.dim, m->hmod));
    {
      HeadStep hs{};
      hs.dt = t1 - t;
      hs.t = t;
      hs.w = so.w;
      hs.uncond_rows = so.guided ? n * m->P : 0;
      if (so.sde_a > 0.f) {
        // App. A.1: sigma_t = a sqrt(t / (1 - t)), evaluated at t' when t = 1
        const double td = t, te = td >= 1.0 ? (double)t1 : td;
        const double sig = so.sde_a * std::sqrt(te / (1.0 - te));
        hs.sde_c = (float)(sig * sig / (2.0 * td));
        hs.nscale = (float)(sig * std::sqrt(std::fabs((double)t1 - td)));
        hs.noise = so.noise + (size_t)k * zn;
      }
      KTimer kt(m, FB_K_HEAD, 2.0 * M * (double)c.dim * m->PD,
                2.0 * M * (double)c.dim + 8.0 * M * m->PD, m->vbuf ? 2 : 1);
      if (m->vbuf) {
        // tensor cores: v = a W_h^T + b_h over npad zero-padded outputs, then the step
        const GemmArgs g = gemm_args(M, m->npad, c.dim, m->act, m->head_wp, m->head_bp, EPI_RESID,
                                     m->vbuf);
        CK(gemm_tc(g, m->derr, m->num_sms, m->st));
        if (k + 1 < S && m->patch_a) {
          hs.patch_next = m->patch_a;
          hs.emb_next = m->emb;
          hs.t_next = t1;
          hs.freq_dim = c.freq_dim;
        }
        CK(euler_step(m->vbuf, m->npad, n, c.latent_c, c.latent_h, c.latent_w, c.patch, hs, z,
                      m->st));
      } else {
        CK(head_euler(m->act, n, c.latent_c, c.latent_h, c.latent_w, c.patch, m->head_w,
                      m->head_b, c.dim, hs, z, m->st));
      }
    }
  }
  return FB_OK;
}

// Byte offset of the contributions in a cached-state buffer (after depth fp32 t values).
size_t state_header_bytes(const fb_cfg& c) { return ((size_t)c.depth * 4 + 255) / 256 * 256; }

fb_status run_sampler(fb_model* m, float* latents, int n, const float* text_ctx,
                      const float* sched, int S, const Plan& plan,
                      const fb_sampler_opts* opts) {
  const fb_cfg& c = m->c;
  const size_t zn = (size_t)n * c.latent_c * c.latent_h * c.latent_w;
  SampOpts so;
  if (opts) {
    so.guided = opts->text_uncond != nullptr;
    so.w = opts->guidance;
    so.sde_a = opts->sde_a;
    if (!(std::isfinite(so.w)) || !(so.sde_a >= 0.f) || !std::isfinite(so.sde_a))
      return fail(FB_EINVAL, "guidance must be finite and sde_a >= 0");
    if (so.sde_a > 0.f && !opts->noise) return fail(FB_EINVAL, "sde_a > 0 needs noise");
    if (so.guided && 2 * n > c.max_n)
      return fail(FB_EINVAL, "guidance needs 2n <= max_n (n=%d, max_n=%d)", n, c.max_n);
  }
  if (so.guided && !m->kvctx_u)
    CKS(dalloc_t(m, &m->kvctx_u, (size_t)c.depth * c.text_len * 2 * c.dim));
  if (so.sde_a > 0.f) {
    if (is_device_ptr(opts->noise)) {
      so.noise = opts->noise;
    } else {
      const size_t ne = zn * S;
      if (ne > m->noise_elems) {
        CK(cudaStreamSynchronize(m->st));
        if (m->noise) {
          cudaFree(m->noise);
          m->allocs.erase(std::find(m->allocs.begin(), m->allocs.end(), (void*)m->noise));
          m->noise = nullptr;
          m->noise_elems = 0;
        }
        CKS(dalloc_t(m, &m->noise, ne));
        m->noise_elems = ne;
      }
      fb_stream_op_not_kernel();
      CK(cudaMemcpyAsync(m->noise, opts->noise, ne * sizeof(float), cudaMemcpyHostToDevice,
                         m->st));
      so.noise = m->noise;
    }
  }
  CKS(begin_call(m));
  // from here on the contribution cache is rewritten: a kept state stays valid only if
  // this call keeps a new one
  m->state_valid = false;
  if (!plan.warm_src.empty()) {
    // warm start: each held layer's contribution into its slot (Plan::warm_src)
    CKS(ensure_anchors(m, (size_t)m->P * c.dim * plan.n_slots));
    const size_t hb = state_header_bytes(c), pd = (size_t)m->P * c.dim;
    for (int l = 0; l < c.depth; ++l) {
      const int sl = plan.warm_src[l];
      if (sl < 0) continue;
      CKS(wait_slot(m, sl, pd));
      fb_stream_op_not_kernel();
      CK(cudaMemcpyAsync(m->anchors + (size_t)sl * pd,
                         static_cast<const uint8_t*>(opts->state) + hb + (size_t)l * pd * 2,
                         pd * 2, cudaMemcpyDefault, m->st));
    }
  }
  CKS(encode_text(m, text_ctx, m->kvctx));
  if (so.guided) CKS(encode_text(m, opts->text_uncond, m->kvctx_u));
  const bool dev = is_device_ptr(latents);
  float* z = dev ? latents : m->zbuf;
  if (!dev) {
    CK(cudaMemcpyAsync(z, latents, zn * sizeof(float), cudaMemcpyHostToDevice, m->st));
    fb_stream_op_not_kernel();
  }
  CKS(sample(m, z, n, sched, S, plan, so));
  if (!dev) {
    fb_stream_op_not_kernel();
    CK(cudaMemcpyAsync(latents, z, zn * sizeof(float), cudaMemcpyDeviceToHost, m->st));
  }
  const fb_status st = end_call(m);
  if (st == FB_OK && !plan.keep_slot.empty()) {
    m->state_valid = true;
    m->state_n = n;
    m->state_nr = so.guided ? 2 * n : n;
    m->state_slot = plan.keep_slot;
    m->state_tau = plan.keep_tau;
  }
  return st;
}

}  // namespace

// =====================================================================================
// C-ABI
// =====================================================================================
extern "C" {

const char* fb_last_error(void) { return g_last_error.c_str(); }

fb_status fb_weights_count(const fb_cfg* cfg, int* count, size_t* total) {
  CKS(check_cfg(cfg));
  if (!count || !total) return fail(FB_EINVAL, "null output pointer");
  auto t = weight_table(*cfg);
  *count = (int)t.size();
  size_t s = 0;
  for (auto& e : t) s += e.numel;
  *total = s;
  return FB_OK;
}

fb_status fb_weights_entry(const fb_cfg* cfg, int idx, const char** name, size_t* offset,
                           size_t* numel) {
  CKS(check_cfg(cfg));
  static thread_local std::vector<WEntry> cache;
  cache = weight_table(*cfg);
  if (idx < 0 || idx >= (int)cache.size()) return fail(FB_EINVAL, "entry %d out of range", idx);
  size_t off = 0;
  for (int i = 0; i < idx; ++i) off += cache[i].numel;
  if (name) *name = cache[idx].name.c_str();
  if (offset) *offset = off;
  if (numel) *numel = cache[idx].numel;
  return FB_OK;
}

void fb_free(fb_model* m) {
  if (!m) return;
  if (m->st) cudaStreamSynchronize(m->st);
  for (auto& p : m->pending) { cudaEventDestroy(p.a); cudaEventDestroy(p.b); }
  for (auto e : m->ev_pool) cudaEventDestroy(e);
  if (m->copy_st) cudaStreamSynchronize(m->copy_st);
  for (auto e : m->slot_ev)
    if (e) cudaEventDestroy(e);
  if (m->copy_st) cudaStreamDestroy(m->copy_st);
  for (void* p : m->allocs) cudaFree(p);
  if (m->herr) cudaFreeHost(m->herr);
  if (m->own) cudaStreamDestroy(m->own);
  delete m;
}

fb_status fb_init_model(const fb_cfg* cfg, const float* weights_host, fb_model** out) {
  if (!out) return fail(FB_EINVAL, "out is NULL");
  *out = nullptr;
  CKS(check_cfg(cfg));
  if (!weights_host) return fail(FB_EINVAL, "weights_host is NULL");
  fb_model* m = new fb_model();
  m->c = *cfg;
  const fb_cfg& c = m->c;
  m->gh = c.latent_h / c.patch;
  m->gw = c.latent_w / c.patch;
  m->P = m->gh * m->gw;
  m->PD = c.latent_c * c.patch * c.patch;
  m->Mmax = (size_t)c.max_n * m->P;
  memset(m->stats, 0, sizeof m->stats);
  auto bail = [&](fb_status s) { fb_free(m); return s; };
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&m->num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return bail(fail(FB_ECUDA, "no CUDA device"));
  }
  m->dev = dev;
  // A blocking stream: its work is ordered after work the caller put on the legacy
  // default stream (e.g. copies that fill the input buffers) and vice versa.
  if (cudaStreamCreateWithFlags(&m->own, cudaStreamDefault) != cudaSuccess)
    return bail(fail(FB_ECUDA, "cudaStreamCreate failed"));
  m->st = m->own;
  if (cudaMallocHost(&m->herr, sizeof(int)) != cudaSuccess)
    return bail(fail(FB_ENOMEM, "cudaMallocHost failed"));

  // weights: matrices bf16, vectors fp32 (all per-layer tables first, contiguous)
  auto table = weight_table(c);
  size_t nmat = 0, nvec = (size_t)c.depth * 6 * c.dim;
  for (auto& e : table)
    if (e.kind == W_MAT) nmat += e.numel;
    else if (e.name.find(".table") == std::string::npos || e.name == "head.table") nvec += e.numel;
  fb_status s;
  if ((s = dalloc(m, &m->wmat, nmat * 2)) != FB_OK) return bail(s);
  if ((s = dalloc(m, &m->wvec, nvec * 4)) != FB_OK) return bail(s);
  float* stage = nullptr;
  size_t max_mat = 0;
  for (auto& e : table) if (e.kind == W_MAT) max_mat = std::max(max_mat, e.numel);
  if ((s = dalloc_t(m, &stage, max_mat)) != FB_OK) return bail(s);
  m->tables = reinterpret_cast<float*>(m->wvec);
  std::map<std::string, void*> ptr;
  size_t off = 0, mo = 0, vo = (size_t)c.depth * 6 * c.dim;
  for (auto& e : table) {
    const float* src = weights_host + off;
    off += e.numel;
    void* dst;
    if (e.kind == W_MAT) {
      dst = reinterpret_cast<bf16*>(m->wmat) + mo;
      mo += e.numel;
      fb_stream_op_not_kernel();
      if (cudaMemcpyAsync(stage, src, e.numel * 4, cudaMemcpyDefault, m->st) != cudaSuccess ||
          f32_to_bf16(stage, reinterpret_cast<bf16*>(dst), e.numel, m->st) != cudaSuccess ||
          cudaStreamSynchronize(m->st) != cudaSuccess)
        return bail(fail(FB_ECUDA, "weight upload failed (%s)", e.name.c_str()));
    } else {
      if (e.name.size() > 6 && e.name.compare(0, 7, "blocks.") == 0 &&
          e.name.find(".table") != std::string::npos) {
        const int l = atoi(e.name.c_str() + 7);
        dst = m->tables + (size_t)l * 6 * c.dim;
      } else {
        dst = reinterpret_cast<float*>(m->wvec) + vo;
        vo += e.numel;
      }
      if (cudaMemcpyAsync(dst, src, e.numel * 4, cudaMemcpyDefault, m->st) != cudaSuccess)
        return bail(fail(FB_ECUDA, "weight upload failed (%s)", e.name.c_str()));
    }
    ptr[e.name] = dst;
  }
  if (cudaStreamSynchronize(m->st) != cudaSuccess) return bail(fail(FB_ECUDA, "weight upload"));
  cudaFree(stage);
  m->allocs.erase(std::find(m->allocs.begin(), m->allocs.end(), (void*)stage));
  auto B = [&](const std::string& n) { return reinterpret_cast<bf16*>(ptr[n]); };
  auto Fp = [&](const std::string& n) { return reinterpret_cast<float*>(ptr[n]); };
  m->patch_w = B("patch.w"); m->patch_b = Fp("patch.b");
  m->time_w1 = B("time.w1"); m->time_b1 = Fp("time.b1");
  m->time_w2 = B("time.w2"); m->time_b2 = Fp("time.b2");
  m->mod_w = B("mod.w"); m->mod_b = Fp("mod.b");
  m->text_w1 = B("text.w1"); m->text_b1 = Fp("text.b1");
  m->text_w2 = B("text.w2"); m->text_b2 = Fp("text.b2");
  m->head_table = Fp("head.table"); m->head_w = B("head.w"); m->head_b = Fp("head.b");
  m->L.resize(c.depth);
  for (int l = 0; l < c.depth; ++l) {
    const std::string p = "blocks." + std::to_string(l) + ".";
    Layer& w = m->L[l];
    w.table = Fp(p + "table");
    w.wqkv = B(p + "attn.wqkv"); w.bqkv = Fp(p + "attn.bqkv");
    w.nq = Fp(p + "attn.norm_q"); w.nk = Fp(p + "attn.norm_k");
    w.wo = B(p + "attn.wo"); w.bo = Fp(p + "attn.bo");
    w.n3w = Fp(p + "norm3.w"); w.n3b = Fp(p + "norm3.b");
    w.cq = B(p + "cross.wq"); w.cbq = Fp(p + "cross.bq");
    w.ckv = B(p + "cross.wkv"); w.cbkv = Fp(p + "cross.bkv");
    w.cnq = Fp(p + "cross.norm_q"); w.cnk = Fp(p + "cross.norm_k");
    w.co = B(p + "cross.wo"); w.cbo = Fp(p + "cross.bo");
    w.w1 = B(p + "ffn.w1"); w.b1 = Fp(p + "ffn.b1");
    w.w2 = B(p + "ffn.w2"); w.b2 = Fp(p + "ffn.b2");
  }

  // activation buffers
  const size_t M = m->Mmax, D = c.dim;
  const size_t zn = (size_t)c.max_n * c.latent_c * c.latent_h * c.latent_w;
  if ((s = dalloc_t(m, &m->hA, M * D)) || (s = dalloc_t(m, &m->hB, M * D)) ||
      (s = dalloc_t(m, &m->act, M * D)) || (s = dalloc_t(m, &m->qkv, M * 3 * D)) ||
      (s = dalloc_t(m, &m->ao, M * D)) || (s = dalloc_t(m, &m->cqb, M * D)) ||
      (s = dalloc_t(m, &m->ffh, M * c.ffn)) ||
      (s = dalloc_t(m, &m->ctx_f, (size_t)c.text_len * c.text_dim)) ||
      (s = dalloc_t(m, &m->ctx_b, (size_t)c.text_len * c.text_dim)) ||
      (s = dalloc_t(m, &m->ctx_h, (size_t)c.text_len * D)) ||
      (s = dalloc_t(m, &m->ctx_p, (size_t)c.text_len * D)) ||
      (s = dalloc_t(m, &m->kvctx, (size_t)c.depth * c.text_len * 2 * D)) ||
      (s = dalloc_t(m, &m->emb, (size_t)c.freq_dim)) || (s = dalloc_t(m, &m->th1, D)) ||
      (s = dalloc_t(m, &m->temb, D)) || (s = dalloc_t(m, &m->mod, 6 * D)) ||
      (s = dalloc_t(m, &m->modl, (size_t)c.depth * 6 * D)) || (s = dalloc_t(m, &m->hmod, 2 * D)) ||
      (s = dalloc_t(m, &m->rope, (size_t)m->P * c.head_dim / 2)) ||
      (s = dalloc_t(m, &m->zbuf, zn)) || (s = dalloc_t(m, &m->derr, 1)))
    return bail(s);
  m->dev_sms = m->num_sms;
  m->sk_clusters = m->num_sms / 2;
  if ((s = dalloc_t(m, &m->sk_ws, (size_t)m->sk_clusters * SK_WS_FLOATS_PER_CLUSTER)) ||
      (s = dalloc_t(m, &m->sk_ctr, (size_t)m->sk_clusters * SK_CTR_PER_CLUSTER)))
    return bail(s);
  if (cudaMemset(m->sk_ctr, 0, (size_t)m->sk_clusters * SK_CTR_PER_CLUSTER * sizeof(int)) !=
      cudaSuccess)
    return bail(fail(FB_ECUDA, "cudaMemset failed"));
  if (m->PD % 64 == 0 && D % 128 == 0) {
    const size_t PDs = m->PD;
    m->npad = (m->PD + 127) / 128 * 128;
    if ((s = dalloc_t(m, &m->patch_a, M * PDs)) ||
        (s = dalloc_t(m, &m->head_wp, (size_t)m->npad * D)) ||
        (s = dalloc_t(m, &m->head_bp, (size_t)m->npad)) ||
        (s = dalloc_t(m, &m->vbuf, M * m->npad)))
      return bail(s);
    if (cudaMemset(m->head_wp, 0, (size_t)m->npad * D * sizeof(bf16)) != cudaSuccess ||
        cudaMemset(m->head_bp, 0, (size_t)m->npad * sizeof(float)) != cudaSuccess ||
        cudaMemcpy(m->head_wp, m->head_w, PDs * D * sizeof(bf16), cudaMemcpyDeviceToDevice) !=
            cudaSuccess ||
        cudaMemcpy(m->head_bp, m->head_b, PDs * sizeof(float), cudaMemcpyDeviceToDevice) !=
            cudaSuccess)
      return bail(fail(FB_ECUDA, "head weight padding failed"));
  }
  // RoPE table: pair j of a head rotates by the token's row (j < head_dim/4) or column,
  // with frequency theta^(-2 j' / (head_dim/2)), j' = j mod head_dim/4.
  {
    const int half = c.head_dim / 2, npair = half / 2;
    std::vector<float2> tab((size_t)m->P * half);
    for (int tok = 0; tok < m->P; ++tok) {
      const int r = tok / m->gw, col = tok % m->gw;
      for (int j = 0; j < half; ++j) {
        const int jj = j % npair;
        const double pos = j < npair ? r : col;
        const double ang = pos * std::pow((double)c.rope_theta, -2.0 * jj / half);
        tab[(size_t)tok * half + j] = make_float2((float)std::cos(ang), (float)std::sin(ang));
      }
    }
    if (cudaMemcpy(m->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice) !=
        cudaSuccess)
      return bail(fail(FB_ECUDA, "rope table upload failed"));
  }
  if (cudaMemset(m->derr, 0, sizeof(int)) != cudaSuccess)
    return bail(fail(FB_ECUDA, "cudaMemset failed"));
  *out = m;
  return FB_OK;
}

fb_status fb_set_stream(fb_model* m, void* stream) {
  if (!m) return fail(FB_EINVAL, "model is NULL");
  CK(cudaStreamSynchronize(m->st));
  m->st = stream ? reinterpret_cast<cudaStream_t>(stream) : m->own;
  fb_stream_op_not_kernel();
  return FB_OK;
}

fb_status fb_set_sm_budget(fb_model* m, int n_sms) {
  if (!m) return fail(FB_EINVAL, "model is NULL");
  if (n_sms == 0) n_sms = m->dev_sms;
  if (n_sms < 2 || n_sms > m->dev_sms)
    return fail(FB_EINVAL, "n_sms=%d outside [2, %d]", n_sms, m->dev_sms);
  CK(cudaStreamSynchronize(m->st));
  m->num_sms = n_sms;
  return FB_OK;
}

fb_status fb_encode_text(fb_model* m, const float* text_ctx) {
  if (!m || !text_ctx) return fail(FB_EINVAL, "null argument");
  CKS(begin_call(m));
  CKS(encode_text(m, text_ctx, m->kvctx));
  return end_call(m);
}

fb_status fb_draft(fb_model* m, float* latents, int n, const float* text_ctx,
                   const float* schedule, int n_steps, const uint8_t* skip_mask,
                   const int32_t* proxy_plan) {
  return fb_draft_ex(m, latents, n, text_ctx, schedule, n_steps, skip_mask, proxy_plan, nullptr);
}

fb_status fb_draft_ex(fb_model* m, float* latents, int n, const float* text_ctx,
                      const float* schedule, int n_steps, const uint8_t* skip_mask,
                      const int32_t* proxy_plan, const fb_sampler_opts* opts) {
  if (!m) return fail(FB_EINVAL, "model is NULL");
  if (n < 0 || n > m->c.max_n) return fail(FB_EINVAL, "n=%d outside [0, max_n=%d]", n, m->c.max_n);
  if (n_steps < 0) return fail(FB_EINVAL, "n_steps < 0");
  if (n == 0 || n_steps == 0) return FB_OK;
  if (!latents || !text_ctx) return fail(FB_EINVAL, "null latents or text_ctx");
  CKS(check_schedule(schedule, n_steps));
  Plan plan;
  CKS(analyse_plan(m->c, schedule, n_steps, skip_mask, proxy_plan, &plan,
                   opts && opts->keep_state));
  return run_sampler(m, latents, n, text_ctx, schedule, n_steps, plan, opts);
}

fb_status fb_refine(fb_model* m, float* latent, const float* text_ctx,
                    const float* full_schedule, int n_steps) {
  return fb_refine_ex(m, latent, text_ctx, full_schedule, n_steps, nullptr);
}

fb_status fb_refine_ex(fb_model* m, float* latent, const float* text_ctx,
                       const float* full_schedule, int n_steps, const fb_sampler_opts* opts) {
  if (!m) return fail(FB_EINVAL, "model is NULL");
  if (n_steps < 0) return fail(FB_EINVAL, "n_steps < 0");
  if (n_steps == 0) return FB_OK;
  if (!latent || !text_ctx) return fail(FB_EINVAL, "null latent or text_ctx");
  CKS(check_schedule(full_schedule, n_steps));
  Plan plan;
  if (opts && opts->state && opts->warm_steps > 0) {
    // §4.2 Stage 3 warm start from a cached state: read its per-layer t (NaN: no Delta)
    if (opts->text_uncond) return fail(FB_EINVAL, "a cached state warm-starts an unguided refine");
    const int L = m->c.depth;
    std::vector<float> tau(L);
    if (is_device_ptr(opts->state)) {
      CK(cudaMemcpy(tau.data(), opts->state, L * sizeof(float), cudaMemcpyDeviceToHost));
    } else {
      std::memcpy(tau.data(), opts->state, L * sizeof(float));
    }
    std::vector<int> slot_of(L, -1);
    int held = 0;
    for (int l = 0; l < L; ++l)
      if (!std::isnan(tau[l])) slot_of[l] = held++;
    warm_plan(L, n_steps, opts->warm_steps, slot_of, &plan);
  } else {
    if (opts && opts->warm_steps < 0) return fail(FB_EINVAL, "warm_steps < 0");
    CKS(analyse_plan(m->c, full_schedule, n_steps, nullptr, nullptr, &plan));
  }
  return run_sampler(m, latent, 1, text_ctx, full_schedule, n_steps, plan, opts);
}

fb_status fb_state_bytes(const fb_model* m, size_t* bytes) {
  if (!m || !bytes) return fail(FB_EINVAL, "null argument");
  *bytes = state_header_bytes(m->c) + (size_t)m->c.depth * m->P * m->c.dim * 2;
  return FB_OK;
}

fb_status fb_state_offload(fb_model* m, int first, int count, void* const* dst) {
  if (!m || !dst) return fail(FB_EINVAL, "null argument");
  if (!m->state_valid) return fail(FB_ESTATE, "no cached state: draft with keep_state first");
  if (first < 0 || count < 1 || first + count > m->state_n)
    return fail(FB_EINVAL, "candidates [%d, %d) outside [0, %d)", first, first + count,
                m->state_n);
  for (int j = 0; j < count; ++j)
    if (!dst[j]) return fail(FB_EINVAL, "dst[%d] is NULL", j);
  const fb_cfg& c = m->c;
  const int L = c.depth;
  if (!m->copy_st) CK(cudaStreamCreateWithFlags(&m->copy_st, cudaStreamNonBlocking));
  const size_t hb = state_header_bytes(c), pd = (size_t)m->P * c.dim;
  const size_t slot_elems = (size_t)m->state_nr * pd;
  const int n_slots = (int)(m->anchor_elems / slot_elems);
  if ((int)m->slot_ev.size() < n_slots) {
    const size_t old = m->slot_ev.size();
    m->slot_ev.resize(n_slots, nullptr);
    m->slot_pending.resize(n_slots, 0);
    for (size_t i = old; i < m->slot_ev.size(); ++i)
      CK(cudaEventCreateWithFlags(&m->slot_ev[i], cudaEventDisableTiming));
  }
  if (m->pending_elems != slot_elems) {
    // copies issued under another slot geometry: let them finish before mixing
    CK(cudaStreamSynchronize(m->copy_st));
    std::fill(m->slot_pending.begin(), m->slot_pending.end(), 0);
    m->pending_elems = slot_elems;
  }
  // the copies start once the work queued so far on the model's stream is done
  cudaEvent_t ready = nullptr;
  CK(cudaEventCreateWithFlags(&ready, cudaEventDisableTiming));
  fb_stream_op_not_kernel();
  CK(cudaEventRecord(ready, m->st));
  CK(cudaStreamWaitEvent(m->copy_st, ready, 0));
  CK(cudaEventDestroy(ready));
  std::vector<uint8_t> hdr(hb, 0);
  std::memcpy(hdr.data(), m->state_tau.data(), L * sizeof(float));
  std::vector<char> dev(count);
  for (int j = 0; j < count; ++j) {
    dev[j] = is_device_ptr(dst[j]);
    if (dev[j]) CK(cudaMemcpyAsync(dst[j], hdr.data(), hb, cudaMemcpyHostToDevice, m->copy_st));
    else std::memcpy(dst[j], hdr.data(), hb);
  }
  for (int l = 0; l < L; ++l) {
    const int sl = m->state_slot[l];
    for (int j = 0; j < count; ++j) {
      uint8_t* out = static_cast<uint8_t*>(dst[j]) + hb + (size_t)l * pd * 2;
      if (sl < 0) {
        if (dev[j]) CK(cudaMemsetAsync(out, 0, pd * 2, m->copy_st));
        else std::memset(out, 0, pd * 2);
        continue;
      }
      CK(cudaMemcpyAsync(out, m->anchors + (size_t)sl * slot_elems + (size_t)(first + j) * pd,
                         pd * 2, cudaMemcpyDefault, m->copy_st));
    }
    if (sl >= 0) {
      CK(cudaEventRecord(m->slot_ev[sl], m->copy_st));
      m->slot_pending[sl] = 1;
    }
  }
  return FB_OK;
}

fb_status fb_state_wait(fb_model* m) {
  if (!m) return fail(FB_EINVAL, "model is NULL");
  if (m->copy_st) CK(cudaStreamSynchronize(m->copy_st));
  std::fill(m->slot_pending.begin(), m->slot_pending.end(), 0);
  return FB_OK;
}

fb_status fb_plan_from_phi(int S, int S_prime, int n_skip, int l_start, int l_end, int f_full,
                           int order, int depth, uint8_t* skip_mask, int32_t* proxy_plan) {
  if (!skip_mask || !proxy_plan) return fail(FB_EINVAL, "null output arrays");
  if (depth < 1 || S_prime < 1 || S_prime > S || f_full < 1 || n_skip < 0 || l_start < 1 ||
      l_start > l_end || l_end > depth || order < 0 || order > 2 || S_prime > 0xFFFF)
    return fail(FB_EINVAL, "invalid phi");
  for (int k = 0; k < S_prime; ++k) {
    const bool full = (k % f_full) == 0;
    const int last_full = k - k % f_full;
    for (int l = 0; l < depth; ++l) {
      const bool sk = k >= n_skip && l >= l_start - 1 && l <= l_end - 1;
      skip_mask[(size_t)k * depth + l] = sk ? 1 : 0;
      proxy_plan[(size_t)k * depth + l] = (sk || full) ? -1 : (last_full | (order << 16));
    }
  }
  return FB_OK;
}

fb_status fb_block_forward(fb_model* m, int layer, float* h, int n, float t) {
  if (!m || !h) return fail(FB_EINVAL, "null argument");
  if (layer < 0 || layer >= m->c.depth) return fail(FB_EINVAL, "layer %d out of range", layer);
  if (n < 0 || n > m->c.max_n) return fail(FB_EINVAL, "n=%d outside [0, max_n]", n);
  if (!m->text_ready) return fail(FB_ESTATE, "fb_encode_text has not been called");
  if (n == 0) return FB_OK;
  if (!is_device_ptr(h)) return fail(FB_EINVAL, "h must be device memory");
  CKS(begin_call(m));
  CKS(time_embed(m, t));
  CKS(block_forward(m, layer, h, n, nullptr));
  return end_call(m);
}

fb_status fb_set_timing(fb_model* m, int mask) {
  if (!m) return fail(FB_EINVAL, "model is NULL");
  m->timing_mask = (unsigned)mask;
  return FB_OK;
}

fb_status fb_get_stats(fb_model* m, fb_kstat* out) {
  if (!m || !out) return fail(FB_EINVAL, "null argument");
  CK(cudaStreamSynchronize(m->st));
  collect_timings(m);
  memcpy(out, m->stats, sizeof m->stats);
  return FB_OK;
}

fb_status fb_reset_stats(fb_model* m) {
  if (!m) return fail(FB_EINVAL, "model is NULL");
  CK(cudaStreamSynchronize(m->st));
  collect_timings(m);
  memset(m->stats, 0, sizeof m->stats);
  return FB_OK;
}

const char* fb_kernel_name(int kind) {
  static const char* names[FB_K_COUNT] = {"gemm_tc", "gemm_simt", "attn_self", "attn_cross",
                                          "ln_mod", "qk_norm_rope", "proxy_add", "patch_embed",
                                          "head_euler", "small"};
  return (kind >= 0 && kind < FB_K_COUNT) ? names[kind] : "?";
}

fb_status fb_op_gemm(fb_model* m, int M, int N, int K, const void* A, const void* W,
                     const float* bias, int epi, void* out, const float* resid,
                     const float* gate, const float* base, void* delta, int impl) {
  if (!m || !A || !W || !out) return fail(FB_EINVAL, "null argument");
  if (M < 1 || N < 1 || K < 1 || epi < 0 || epi > 3) return fail(FB_EINVAL, "bad sizes / epi");
  if (epi == EPI_RESID_DELTA && !resid) return fail(FB_EINVAL, "resid required");
  if (epi == EPI_RESID_DELTA && (!base || !delta)) return fail(FB_EINVAL, "base/delta required");
  if (N % 8) return fail(FB_EINVAL, "N must be a multiple of 8");
  GemmArgs g = gemm_args(M, N, K, (const bf16*)A, (const bf16*)W, bias, epi, out);
  g.epi.resid = resid;
  g.epi.gate = gate;
  g.epi.base = base;
  g.epi.delta = (bf16*)delta;
  CKS(begin_call(m));
  if (impl < 0 || impl > 4) return fail(FB_EINVAL, "impl must be 0 .. 4");
  for (int r = 0; r < m->op_repeat; ++r) CKS(run_gemm(m, g, impl));
  return end_call(m);
}

fb_status fb_op_attention(fb_model* m, const void* Q, int ldq, const void* K, int ldk,
                          const void* V, int ldv, void* O, int ldo, int batch, int Lq, int Lkv,
                          int kv_batch_rows, int heads, int head_dim, int impl) {
  if (!m || !Q || !K || !V || !O) return fail(FB_EINVAL, "null argument");
  if (impl < 0 || impl > 4) return fail(FB_EINVAL, "impl must be 0 .. 4");
  if (batch < 1 || Lq < 1 || Lkv < 1 || heads < 1 || (head_dim != 64 && head_dim != 128))
    return fail(FB_EINVAL, "bad sizes");
  AttnArgs a{};
  a.Q = (const bf16*)Q; a.K = (const bf16*)K; a.V = (const bf16*)V; a.O = (bf16*)O;
  a.ldq = ldq; a.ldk = ldk; a.ldv = ldv; a.ldo = ldo;
  a.batch = batch; a.Lq = Lq; a.Lkv = Lkv; a.kv_batch_rows = kv_batch_rows;
  a.heads = heads; a.head_dim = head_dim;
  CKS(begin_call(m));
  for (int r = 0; r < m->op_repeat; ++r) CKS(run_attn(m, a, FB_K_ATTN_SELF, impl));
  return end_call(m);
}

}  // extern "C"

// ---- allocation-free stream-K GEMM --------------------------------------------------
namespace {
// Static device state of fb_gemm_streamk_noalloc: partials for FB_NOALLOC_MAX_PAIRS SM
// pairs, their per-tile counters (zero at load, left zero by every launch) and an error
// word. Shared by all calls on a device, so overlapping calls race.
static __device__ __align__(256) float g_na_ws[FB_NOALLOC_MAX_PAIRS * SK_WS_FLOATS_PER_CLUSTER];
static __device__ __align__(256) int g_na_ctr[FB_NOALLOC_MAX_PAIRS * SK_CTR_PER_CLUSTER];
static __device__ __align__(256) int g_na_err[1];

struct NoAllocDev {
  bool ready = false;
  float* ws = nullptr;
  int* ctr = nullptr;
  int* err = nullptr;
  int num_sms = 0;
};
constexpr int kNoAllocDevices = 64;
NoAllocDev g_na_dev[kNoAllocDevices];
std::mutex g_na_mu;

// Symbol addresses and SM count of the current device, looked up once per device.
fb_status noalloc_setup(NoAllocDev** out) {
  int dev = 0;
  CK(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kNoAllocDevices) return fail(FB_EINVAL, "device %d out of range", dev);
  std::lock_guard<std::mutex> lock(g_na_mu);
  NoAllocDev& d = g_na_dev[dev];
  if (!d.ready) {
    CK(cudaGetSymbolAddress(reinterpret_cast<void**>(&d.ws), g_na_ws));
    CK(cudaGetSymbolAddress(reinterpret_cast<void**>(&d.ctr), g_na_ctr));
    CK(cudaGetSymbolAddress(reinterpret_cast<void**>(&d.err), g_na_err));
    CK(cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev));
    d.ready = true;
  }
  *out = &d;
  return FB_OK;
}
}  // namespace

extern "C" {

fb_status fb_gemm_streamk_noalloc(void* stream, int M, int N, int K, const void* A,
                                  const void* W, const float* bias, int epi, void* out,
                                  const float* resid, const float* gate, const float* base,
                                  void* delta) {
  if (!A || !W || !out) return fail(FB_EINVAL, "null argument");
  if (M < 1 || N < 1 || K < 1 || epi < 0 || epi > 3) return fail(FB_EINVAL, "bad sizes / epi");
  if (epi == EPI_RESID_DELTA && !resid) return fail(FB_EINVAL, "resid required");
  if (epi == EPI_RESID_DELTA && (!base || !delta)) return fail(FB_EINVAL, "base/delta required");
  if (N % 256) return fail(FB_EINVAL, "N must be a multiple of 256");
  GemmArgs g = gemm_args(M, N, K, (const bf16*)A, (const bf16*)W, bias, epi, out);
  g.epi.resid = resid;
  g.epi.gate = gate;
  g.epi.base = base;
  g.epi.delta = (bf16*)delta;
  if (!gemm_tc_supported(g)) return fail(FB_EINVAL, "shape or alignment not supported");
  NoAllocDev* d = nullptr;
  CKS(noalloc_setup(&d));
  const int pairs = d->num_sms / 2;
  if (pairs > FB_NOALLOC_MAX_PAIRS)
    return fail(FB_EINVAL, "%d SM pairs: the static workspace holds %d", pairs,
                FB_NOALLOC_MAX_PAIRS);
  const long long units = (long long)((M + 255) / 256) * (N / 256) * (K / 64);
  if (units < 4LL * pairs)
    return fail(FB_EINVAL, "%lld (tile, K block) units: stream-K needs >= %d", units, 4 * pairs);
  g.sk_ws = d->ws;
  g.sk_ctr = d->ctr;
  g.sk_clusters = FB_NOALLOC_MAX_PAIRS;
  g.sk_mode = 2;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  fb_stream_op_not_kernel();
  CK(cudaMemsetAsync(d->err, 0, sizeof(int), st));
  CK(gemm_tc(g, d->err, d->num_sms, st, false));
  int herr = 0;
  fb_stream_op_not_kernel();
  CK(cudaMemcpyAsync(&herr, d->err, sizeof(int), cudaMemcpyDeviceToHost, st));
  CK(cudaStreamSynchronize(st));
  if (herr != 0) {
    CK(cudaMemsetAsync(d->ctr, 0, sizeof(int) * FB_NOALLOC_MAX_PAIRS * SK_CTR_PER_CLUSTER, st));
    CK(cudaStreamSynchronize(st));
    return fail(FB_ECUDA, herr == FB_DEVERR_WAIT_TIMEOUT ? "device wait timed out"
                                                         : "device error %d", herr);
  }
  return FB_OK;
}

fb_status fb_set_op_repeat(fb_model* m, int n) {
  if (!m || n < 1) return fail(FB_EINVAL, "model is NULL or n < 1");
  m->op_repeat = n;
  return FB_OK;
}

fb_status fb_set_device_wait_limit(unsigned long long ns) {
  if (ns == 0) ns = FB_WAIT_LIMIT_NS;
  CK(gemm_tc_set_wait_limit(ns));
  CK(attention_tc_set_wait_limit(ns));
  return FB_OK;
}

fb_status fb_test_fail_alloc(long k) {
  g_fail_at.store(-1);
  g_alloc_calls.store(0);
  g_fail_at.store(k < 0 ? -1 : k);
  return FB_OK;
}

long fb_test_alloc_calls(void) { return g_alloc_calls.load(); }

}  // extern "C"

// Shared frame of the probes below: `n` 64-bit words of output (cycles), an error word and
// a float sink on the device, one launch on the legacy stream, a device synchronisation.
template <typename Launch>
static fb_status run_probe(size_t n, std::vector<unsigned long long>& h, Launch launch) {
  unsigned long long* cyc = nullptr;
  int* err = nullptr;
  float* sink = nullptr;
  if (cudaMalloc(&cyc, n * sizeof(unsigned long long)) != cudaSuccess ||
      cudaMalloc(&err, sizeof(int)) != cudaSuccess || cudaMalloc(&sink, sizeof(float)) != cudaSuccess) {
    cudaFree(cyc);
    cudaFree(err);
    cudaFree(sink);
    cudaGetLastError();
    return fail(FB_ENOMEM, "cudaMalloc failed");
  }
  h.assign(n, 0ull);
  int herr = 0;
  cudaError_t e = cudaMemset(err, 0, sizeof(int));
  if (e == cudaSuccess) e = cudaMemset(cyc, 0, n * sizeof(unsigned long long));
  fb_stream_op_not_kernel();
  if (e == cudaSuccess) e = launch(cyc, err, sink);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e == cudaSuccess)
    e = cudaMemcpy(h.data(), cyc, n * sizeof(unsigned long long), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(&herr, err, sizeof(int), cudaMemcpyDeviceToHost);
  cudaFree(cyc);
  cudaFree(err);
  cudaFree(sink);
  if (e != cudaSuccess) return fail(FB_ECUDA, "probe failed: %s", cudaGetErrorString(e));
  if (herr != 0) return fail(FB_ECUDA, "device wait timed out");
  return FB_OK;
}

static fb_status device_sms(int* sms) {
  int dev = 0;
  CK(cudaGetDevice(&dev));
  CK(cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev));
  return FB_OK;
}

extern "C" {

fb_status fb_probe_mma_gap(int gap, double* mac_per_clk) {
  if (!mac_per_clk || gap < 0 || gap > 100000)
    return fail(FB_EINVAL, "gap 0 .. 100000 clocks, non-NULL output");
  int sms = 0;
  CKS(device_sms(&sms));
  const int batches = 2048;
  std::vector<unsigned long long> h;
  CKS(run_probe(sms, h, [&](unsigned long long* c, int* e, float*) {
    return mma_gap_probe(gap, batches, sms, c, e, nullptr);
  }));
  const unsigned long long slowest = *std::max_element(h.begin(), h.end());
  *mac_per_clk = 128.0 * 128 * 16 * 8.0 * batches / (double)slowest;
  return FB_OK;
}

fb_status fb_probe_mufu(int op, double* per_clk) {
  if (!per_clk || op < 0 || op > 3)
    return fail(FB_EINVAL, "op 0 (ex2), 1 (tanh), 2 (rcp), 3 (ex2 on f16 pairs)");
  int sms = 0;
  CKS(device_sms(&sms));
  const int reps = 4096;
  std::vector<unsigned long long> h;
  CKS(run_probe(sms, h, [&](unsigned long long* c, int*, float* sink) {
    return mufu_probe(op, reps, sms, c, sink, nullptr);
  }));
  const unsigned long long slowest = *std::max_element(h.begin(), h.end());
  *per_clk = 256.0 * 16.0 * reps * (op == 3 ? 2.0 : 1.0) / (double)slowest;
  return FB_OK;
}

fb_status fb_probe_mma_mix(int form, int loaders, int loader_gap, double* mac_per_clk) {
  if (!mac_per_clk || form < 0 || form > 13 || loaders < 0 || loaders > 7 || loader_gap < 0 ||
      loader_gap > 100000)
    return fail(FB_EINVAL, "form 0..13, loaders 0..7, loader_gap 0..100000, non-NULL output");
  int sms = 0;
  CKS(device_sms(&sms));
  const int batches = 1024;
  std::vector<unsigned long long> h;
  CKS(run_probe(sms, h, [&](unsigned long long* c, int* e, float* sink) {
    return mma_mix_probe(form, loaders, loader_gap, batches, sms, c, e, sink, nullptr);
  }));
  const unsigned long long slowest = *std::max_element(h.begin(), h.end());
  const double per_batch = form % 7 >= 3 ? 32.0 : 16.0;
  *mac_per_clk = 128.0 * 128 * 16 * per_batch * batches / (double)slowest;
  return FB_OK;
}

fb_status fb_probe_tmem_load(int busy, double* clocks) {
  if (!clocks) return fail(FB_EINVAL, "non-NULL output");
  int sms = 0;
  CKS(device_sms(&sms));
  std::vector<unsigned long long> h;
  CKS(run_probe((size_t)sms * 4, h, [&](unsigned long long* c, int* e, float* sink) {
    return tmem_load_probe(2000, busy ? 1 : 0, sms, c, e, sink, nullptr);
  }));
  double sum = 0;
  for (unsigned long long v : h) sum += (double)v;
  *clocks = sum / (double)h.size();
  return FB_OK;
}

fb_status fb_probe_mma_rate(int issuers, int n, int reps, double* mac_per_clk) {
  if (!mac_per_clk || issuers < 1 || issuers > 4 || (n != 64 && n != 128 && n != 256) ||
      issuers * n > 512 || reps < 1)
    return fail(FB_EINVAL, "issuers 1..4, n 64/128/256, issuers * n <= 512 TMEM columns, "
                           "reps >= 1, non-NULL output");
  int dev = 0, sms = 0;
  CK(cudaGetDevice(&dev));
  CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  unsigned long long* cyc = nullptr;
  int* err = nullptr;
  CK(cudaMalloc(&cyc, sizeof(unsigned long long) * sms));
  if (cudaMalloc(&err, sizeof(int)) != cudaSuccess) {
    cudaFree(cyc);
    return fail(FB_ENOMEM, "cudaMalloc failed");
  }
  std::vector<unsigned long long> h(sms);
  int herr = 0;
  cudaError_t e = cudaMemset(err, 0, sizeof(int));
  if (e == cudaSuccess) e = cudaMemset(cyc, 0, sizeof(unsigned long long) * sms);
  fb_stream_op_not_kernel();
  if (e == cudaSuccess) e = mma_rate_probe(issuers, n, reps, sms, cyc, err, nullptr);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e == cudaSuccess)
    e = cudaMemcpy(h.data(), cyc, sizeof(unsigned long long) * sms, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(&herr, err, sizeof(int), cudaMemcpyDeviceToHost);
  cudaFree(cyc);
  cudaFree(err);
  if (e != cudaSuccess) return fail(FB_ECUDA, "probe failed: %s", cudaGetErrorString(e));
  if (herr != 0) return fail(FB_ECUDA, "device wait timed out");
  const unsigned long long slowest = *std::max_element(h.begin(), h.end());
  *mac_per_clk = 128.0 * n * 16 * (double)issuers * reps / (double)slowest;
  return FB_OK;
}

fb_status fb_test_poison_counters(fb_model* m) {
  int* ctr = nullptr;
  size_t n = 0;
  cudaStream_t st = nullptr;
  if (m) {
    ctr = m->sk_ctr;
    n = (size_t)m->sk_clusters * SK_CTR_PER_CLUSTER;
    st = m->st;
  } else {
    NoAllocDev* d = nullptr;
    CKS(noalloc_setup(&d));
    ctr = d->ctr;
    n = (size_t)FB_NOALLOC_MAX_PAIRS * SK_CTR_PER_CLUSTER;
  }
  if (!ctr) return fail(FB_EINVAL, "no stream-K counters");
  fb_stream_op_not_kernel();
  CK(cudaMemsetAsync(ctr, 0x80, n * sizeof(int), st));  // every counter 0x80808080 < 0
  CK(cudaStreamSynchronize(st));
  return FB_OK;
}

}  // extern "C"

// ---- draft / refine pipeline step -------------------------------------------------
extern "C" fb_status fb_pipeline_step(fb_model* drafter, float* latents, int n,
                                      const float* text_ctx, const float* draft_schedule,
                                      int n_draft_steps, const uint8_t* skip_mask,
                                      const int32_t* proxy_plan,
                                      const fb_sampler_opts* draft_opts, fb_model* refiner,
                                      float* refine_latent, const float* refine_schedule,
                                      int n_refine_steps,
                                      const fb_sampler_opts* refine_opts) {
  if (!drafter) return fail(FB_EINVAL, "drafter is NULL");
  if (refine_latent && (!refiner || refiner == drafter))
    return fail(FB_EINVAL, "the refine needs its own model");
  // the refine on a worker thread (its own model and stream), the draft on this one;
  // the worker's status and message come back to this thread (errors are per thread)
  fb_status rs = FB_OK;
  std::string rmsg;
  std::thread worker;
  if (refine_latent) {
    worker = std::thread([&] {
      // a new thread starts on device 0: make the refiner's device current first
      const cudaError_t e = cudaSetDevice(refiner->dev);
      if (e != cudaSuccess) {
        rs = FB_ECUDA;
        rmsg = std::string("cudaSetDevice failed: ") + cudaGetErrorString(e);
        return;
      }
      rs = fb_refine_ex(refiner, refine_latent, text_ctx, refine_schedule, n_refine_steps,
                        refine_opts);
      if (rs != FB_OK) rmsg = g_last_error;
    });
  }
  const fb_status ds = fb_draft_ex(drafter, latents, n, text_ctx, draft_schedule,
                                   n_draft_steps, skip_mask, proxy_plan, draft_opts);
  const std::string dmsg = ds != FB_OK ? g_last_error : std::string();
  if (worker.joinable()) worker.join();
  if (ds != FB_OK) return fail(ds, "draft: %s", dmsg.c_str());
  if (rs != FB_OK) return fail(rs, "refine: %s", rmsg.c_str());
  return FB_OK;
}

// ---- SM partitions (green contexts) ------------------------------------------------
// The driver's green-context calls are looked up at run time (as cuTensorMapEncodeTiled
// is), so the library needs no link against the driver library.
struct fb_sm_split {
  CUgreenCtx g[2] = {nullptr, nullptr};
  CUstream s[2] = {nullptr, nullptr};
  int sms[2] = {0, 0};
};

namespace {
template <typename F>
bool drv_fn(const char* name, int version, F* out) {
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &p, version, cudaEnableDefault, &q) !=
          cudaSuccess ||
      q != cudaDriverEntryPointSuccess || !p) {
    cudaGetLastError();
    return false;
  }
  *out = reinterpret_cast<F>(p);
  return true;
}
struct GreenFns {
  decltype(&cuDeviceGetDevResource) get_res = nullptr;
  decltype(&cuDevSmResourceSplitByCount) split = nullptr;
  decltype(&cuDevResourceGenerateDesc) gen_desc = nullptr;
  decltype(&cuGreenCtxCreate) create = nullptr;
  decltype(&cuGreenCtxStreamCreate) stream_create = nullptr;
  decltype(&cuGreenCtxDestroy) destroy = nullptr;
  decltype(&cuStreamDestroy) stream_destroy = nullptr;
  bool ok = false;
};
const GreenFns& green_fns() {
  static const GreenFns f = [] {
    GreenFns g;
    g.ok = drv_fn("cuDeviceGetDevResource", 12040, &g.get_res) &&
           drv_fn("cuDevSmResourceSplitByCount", 12040, &g.split) &&
           drv_fn("cuDevResourceGenerateDesc", 12040, &g.gen_desc) &&
           drv_fn("cuGreenCtxCreate", 12040, &g.create) &&
           drv_fn("cuGreenCtxStreamCreate", 12050, &g.stream_create) &&
           drv_fn("cuGreenCtxDestroy", 12040, &g.destroy) &&
           drv_fn("cuStreamDestroy", 4000, &g.stream_destroy);
    return g;
  }();
  return f;
}
}  // namespace

extern "C" {

void fb_sm_split_free(fb_sm_split* sp) {
  if (!sp) return;
  const GreenFns& f = green_fns();
  for (int i = 0; i < 2; ++i) {
    if (sp->s[i]) {
      cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(sp->s[i]));
      if (f.ok) f.stream_destroy(sp->s[i]);
    }
    if (sp->g[i] && f.ok) f.destroy(sp->g[i]);
  }
  cudaGetLastError();
  delete sp;
}

fb_status fb_sm_split_create(int n_sms, fb_sm_split** out) {
  if (!out) return fail(FB_EINVAL, "out is NULL");
  *out = nullptr;
  const GreenFns& f = green_fns();
  if (!f.ok) return fail(FB_ECUDA, "green contexts are not available from this driver");
  int dev = 0;
  CK(cudaGetDevice(&dev));
  CK(cudaFree(nullptr));  // the device's primary context exists from here on
  CUdevResource all;
  if (f.get_res(static_cast<CUdevice>(dev), &all, CU_DEV_RESOURCE_TYPE_SM) != CUDA_SUCCESS)
    return fail(FB_ECUDA, "cuDeviceGetDevResource failed");
  if (n_sms < 2 || n_sms > (int)all.sm.smCount - 2)
    return fail(FB_EINVAL, "n_sms=%d outside [2, %u]", n_sms, all.sm.smCount - 2);
  CUdevResource parts[2];
  unsigned n_groups = 1;
  if (f.split(&parts[0], &n_groups, &all, &parts[1], 0, (unsigned)n_sms) != CUDA_SUCCESS ||
      n_groups != 1)
    return fail(FB_ECUDA, "cuDevSmResourceSplitByCount failed");
  fb_sm_split* sp = new fb_sm_split;
  for (int i = 0; i < 2; ++i) {
    CUdevResourceDesc desc;
    if (f.gen_desc(&desc, &parts[i], 1) != CUDA_SUCCESS ||
        f.create(&sp->g[i], desc, static_cast<CUdevice>(dev), CU_GREEN_CTX_DEFAULT_STREAM) !=
            CUDA_SUCCESS ||
        f.stream_create(&sp->s[i], sp->g[i], CU_STREAM_NON_BLOCKING, 0) != CUDA_SUCCESS) {
      fb_sm_split_free(sp);
      return fail(FB_ECUDA, "green context %d creation failed", i);
    }
    sp->sms[i] = (int)parts[i].sm.smCount;
  }
  *out = sp;
  return FB_OK;
}

fb_status fb_sm_split_info(const fb_sm_split* sp, int part, void** stream, int* sms) {
  if (!sp || !stream || !sms || part < 0 || part > 1) return fail(FB_EINVAL, "bad argument");
  *stream = reinterpret_cast<void*>(sp->s[part]);
  *sms = sp->sms[part];
  return FB_OK;
}

}  // extern "C"
