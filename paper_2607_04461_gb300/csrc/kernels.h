// Host-side launchers of the sm_103a kernels (internal to libflashbon.so).
// Every launcher enqueues on `st` and returns the cudaError_t of the launch.
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "common.cuh"

// ---- GEMM: out[M][N] = epilogue(A[M][K] * W[N][K]^T) --------------------------------
struct GemmArgs {
  int M, N, K;
  const bf16* A;  // row-major, leading dimension lda
  int lda;
  const bf16* W;  // row-major [N][K], leading dimension ldw
  int ldw;
  int kind;       // EPI_*
  GemmEpi epi;
  // Stream-K workspace of the 2-SM kernel (null: data-parallel tiles only): room for
  // sk_clusters clusters (sk_clusters * 131072 floats) and sk_clusters * 16 counters that
  // start at zero and are left at zero. sk_mode: 0 automatic, 1 never, 2 always.
  float* sk_ws;
  int* sk_ctr;
  int sk_clusters;
  int sk_mode;
};
// floats and counters of the stream-K workspace per cluster
constexpr size_t SK_WS_FLOATS_PER_CLUSTER = 2 * 2 * 8 * 4096;
constexpr int SK_CTR_PER_CLUSTER = 16;
// tcgen05 path: requires N % 128 == 0, K % 64 == 0, 16-byte aligned rows. Uses the
// 2-SM (cta_group::2) kernel when N % 256 == 0 unless force_1sm.
bool gemm_tc_supported(const GemmArgs& g);
cudaError_t gemm_tc(const GemmArgs& g, int* err, int num_sms, cudaStream_t st,
                    bool force_1sm = false);
// Sets the gemm_tc unit's device wait limit on the current device (ns; see common.cuh).
cudaError_t gemm_tc_set_wait_limit(unsigned long long ns);
// CUDA-core path: requires N % 8 == 0.
cudaError_t gemm_simt(const GemmArgs& g, cudaStream_t st);

// ---- attention: O = softmax(Q K^T / sqrt(dh)) V ----------------------------------
struct AttnArgs {
  const bf16 *Q, *K, *V;
  bf16* O;
  int ldq, ldk, ldv, ldo;  // row strides (elements)
  int batch, Lq, Lkv;
  int kv_batch_rows;       // row offset of batch b's K/V (0 = shared)
  int heads, head_dim;
  int tc_variant;          // tcgen05 kernel: 0 automatic, 1 128-query CTAs, 2 256-query CTAs,
                           // 3 the persistent 256-query kernel
  int sms;                 // SMs the launch may use (its choice of CTA size); 0: the device's
};
// mma.sync (warp-level) kernel: head_dim 64 or 128.
cudaError_t attention(const AttnArgs& a, cudaStream_t st);
// tcgen05/TMEM kernel: head_dim 128, 16-byte aligned rows.
bool attention_tc_supported(const AttnArgs& a);
cudaError_t attention_tc(const AttnArgs& a, int* err, cudaStream_t st);
// Sets the attention_tc unit's device wait limit on the current device (ns).
cudaError_t attention_tc_set_wait_limit(unsigned long long ns);

// ---- pointwise / small kernels ------------------------------------------------------
// out[r][:] = bf16(LN(x[r][:]) * (mul_base + mul[:]) + add[:]), x fp32 [rows][D].
cudaError_t ln_mod(const float* x, bf16* out, int rows, int D, float eps, float mul_base,
                   const float* mul, const float* add, cudaStream_t st);
// In place on bf16 rows: x[r][col0 + :D] = RMSNorm(.) * w, then (if rope != null) RoPE
// with table rope[(r % tokens)][head_dim/2] of (cos, sin) per adjacent pair.
// Two segments (col0, w0) and (col1, w1) when nseg == 2.
cudaError_t qk_norm_rope(bf16* x, int rows, int ld, int D, int nseg, int col0, const float* w0,
                         int col1, const float* w1, float eps, const float2* rope,
                         int tokens, int head_dim, cudaStream_t st);
// h[i] += sum_t coef[t] * anchor_t[i] over n_elems fp32 elements (bf16 anchors).
#define FB_PROXY_MAX_TERMS 64
struct ProxyTerms {
  const bf16* ptr[FB_PROXY_MAX_TERMS];
  float coef[FB_PROXY_MAX_TERMS];
  int n;
};
cudaError_t proxy_add(float* h, size_t n_elems, const ProxyTerms& t, cudaStream_t st);
// h[(b*P + tok)][:] = W_p * patch(z_b, tok) + b_p.
cudaError_t patch_embed(const float* z, int n, int C, int H, int W, int p, const bf16* Wp,
                        const float* bp, int D, float* h, cudaStream_t st);
// v = unpatchify(a * Wh^T + bh) from a bf16 [n*P][D]; with guidance (uncond_rows > 0) also
// v_u from rows uncond_rows.. and v = v_u + w (v - v_u). Then the step on z[b]:
//   ODE (noise == null): z += dt v
//   SDE: z += (v + sde_c (z + (1 - t) v)) dt + nscale * noise[b]   (noise like z)
struct HeadStep {
  float dt, t, w, sde_c, nscale;
  int uncond_rows;        // 0: no guidance
  const float* noise;     // null: ODE step
  // euler_step only: the next step's conditioning, written from the updated z (null: last
  // step). patch_next: bf16 patch rows (as patchify writes them); emb_next: the sinusoidal
  // embedding of t_next (as timestep_sincos writes it, freq_dim entries).
  bf16* patch_next;
  float* emb_next;
  float t_next;
  int freq_dim;
};
cudaError_t head_euler(const bf16* a, int n, int C, int H, int W, int p, const bf16* Wh,
                       const float* bh, int D, const HeadStep& hs, float* z, cudaStream_t st);
// out[b P + tok][(ch, dy, dx)] = bf16(z[b][ch][r p + dy][c p + dx]) for token tok = r (W/p) + c:
// the patch rows of z, the A operand of the tensor-core patch embedding (C p p % 8 == 0).
cudaError_t patchify(const float* z, int n, int C, int H, int W, int p, bf16* out,
                     cudaStream_t st);
// The guidance combination and step of head_euler, with v[row][o] (fp32, leading dimension
// ldv >= C p p) the head output a Wh^T + bh computed by the tensor-core GEMM; with
// hs.patch_next / hs.emb_next also the next step's patch rows and timestep embedding
// (C p p % 8 == 0).
cudaError_t euler_step(const float* v, int ldv, int n, int C, int H, int W, int p,
                       const HeadStep& hs, float* z, cudaStream_t st);
// y[o] = act_out(b[o] + sum_k W[o][k] act_in(x[k])), act: 0 none, 1 SiLU.
cudaError_t gemv(const bf16* W, const float* b, const float* x, float* y, int O, int K,
                 int act_in, int act_out, cudaStream_t st);
// emb = [cos(1000 t f_k), sin(1000 t f_k)], f_k = 10000^(-k/half).
cudaError_t timestep_sincos(float t, int dim, float* emb, cudaStream_t st);
// modl[l][j][:] = mod[j][:] + table_l[j][:] (6 rows, all layers); head[j] = htab[j] + temb.
cudaError_t mod_prepare(const float* mod, const float* tables, int L, int D,
                        float* modl, const float* htab, const float* temb, float* head_mod,
                        cudaStream_t st);
cudaError_t f32_to_bf16(const float* x, bf16* y, size_t n, cudaStream_t st);

// ---- measurement probe ----------------------------------------------------------------
// One CTA per entry of `grid`, each timing (SM clock cycles, cycles[cta]) `reps` tcgen05.mma
// kind::f16 instructions of M = 128, K = 16 and width N (64, 128 or 256) issued by each of
// `issuers` warps (1-4) into accumulators of their own.
cudaError_t mma_gap_probe(int gap, int batches, int grid, unsigned long long* cycles, int* err,
                          cudaStream_t st);
cudaError_t mufu_probe(int op, int reps, int grid, unsigned long long* cycles, float* sink,
                       cudaStream_t st);
cudaError_t tmem_load_probe(int reps, int busy, int grid, unsigned long long* cycles, int* err,
                            float* sink, cudaStream_t st);
cudaError_t mma_mix_probe(int form, int loaders, int loader_gap, int batches, int grid,
                          unsigned long long* cycles, int* err, float* sink, cudaStream_t st);
cudaError_t mma_rate_probe(int issuers, int N, int reps, int grid, unsigned long long* cycles,
                           int* err, cudaStream_t st);
