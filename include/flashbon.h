/* flashbon.h -- C-ABI of the GB300 (sm_103a) Flash-BoN draft-generation library.
 *
 * The library runs the hot path of Flash-BoN ("Instant Drafts for Inference-Time
 * Scaling in Diffusion Models"): a pool of N seed-varied candidates is denoised by a
 * DiT flow-matching model under the paper's three acceleration knobs (§4.1):
 * a truncated timestep schedule (early stopping), a per-step layer-skip set (Eq. 6)
 * and activation proxies (Eqs. 3-5) that stand in for a block's computation; then one
 * selected latent is refined with full computation (§4.2, Stage 3).
 *
 * Conventions for every entry point:
 *  - Return an fb_status; they never abort. fb_last_error() gives a message for the
 *    last failing call on the calling thread.
 *  - The caller owns every input and output buffer. The model owns its device weights,
 *    activation buffers and the proxy cache.
 *  - All work is enqueued on the model's stream (fb_set_stream; default: a blocking
 *    stream the model creates, ordered with the legacy default stream, so inputs written
 *    there are complete before the model reads them) and the call returns after that
 *    stream has finished the work. With a caller's stream set, the caller orders its own
 *    writes of the inputs before the call (same stream or an event).
 *  - "host or device" pointers are classified with cudaPointerGetAttributes: device
 *    (or managed) memory is used in place; host memory is staged through device
 *    buffers inside the call.
 *  - A device-side wait that exceeds its time limit (about two seconds) makes the
 *    kernel give up, and the call returns FB_ECUDA with "device wait timed out".
 */
#ifndef FLASHBON_H
#define FLASHBON_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum fb_status {
  FB_OK = 0,
  FB_EINVAL = 1,  /* bad argument: null pointer, size out of range, bad schedule */
  FB_ENOMEM = 2,  /* device or host allocation failed */
  FB_ECUDA = 3,   /* a CUDA call or a kernel failed, or a device wait timed out */
  FB_EPLAN = 4,   /* malformed skip_mask / proxy_plan */
  FB_ESTATE = 5   /* call out of order, e.g. block forward before fb_encode_text */
} fb_status;

/* Model shape. Linear weights are [out][in]. dim = heads * head_dim; head_dim is 64
 * or 128; latent_h and latent_w are multiples of patch; patch_dim =
 * latent_c * patch * patch <= 64. max_n bounds the candidates per call (buffers are
 * sized for max_n * tokens rows). eps_ln: LayerNorm epsilon; eps_rms: RMSNorm epsilon;
 * rope_theta: RoPE base; freq_dim: sinusoidal timestep-embedding width (even). */
typedef struct fb_cfg {
  int depth, dim, heads, head_dim, ffn, text_len, text_dim;
  int latent_c, latent_h, latent_w, patch, max_n, freq_dim;
  float eps_ln, eps_rms, rope_theta;
} fb_cfg;

typedef struct fb_model fb_model;

/* ---- weight layout -------------------------------------------------------------
 * The packed host weight buffer is fp32, tensors back to back in entry order
 * 0..count-1. Entry order and names:
 *   patch.w [D][C p p], patch.b [D], time.w1 [D][freq_dim], time.b1 [D],
 *   time.w2 [D][D], time.b2 [D], mod.w [6D][D], mod.b [6D], text.w1 [D][text_dim],
 *   text.b1 [D], text.w2 [D][D], text.b2 [D], head.table [2][D], head.w [C p p][D],
 *   head.b [C p p], then for each block l = 0..depth-1 with prefix "blocks.<l>.":
 *   table [6][D], attn.wqkv [3D][D], attn.bqkv [3D], attn.norm_q [D],
 *   attn.norm_k [D], attn.wo [D][D], attn.bo [D], norm3.w [D], norm3.b [D],
 *   cross.wq [D][D], cross.bq [D], cross.wkv [2D][D], cross.bkv [2D],
 *   cross.norm_q [D], cross.norm_k [D], cross.wo [D][D], cross.bo [D],
 *   ffn.w1 [F][D], ffn.b1 [F], ffn.w2 [D][F], ffn.b2 [D].
 * fb_weights_entry: name (static string), element offset into the packed buffer and
 * element count of entry idx. FB_EINVAL for idx out of range or a bad cfg. */
fb_status fb_weights_count(const fb_cfg* cfg, int* count, size_t* total_elems);
fb_status fb_weights_entry(const fb_cfg* cfg, int idx, const char** name,
                           size_t* offset, size_t* numel);

/* ---- model --------------------------------------------------------------------
 * fb_init_model: validates cfg, copies the packed fp32 weights to the device as bf16
 * (matrices) and fp32 (biases, norm scales, modulation tables), allocates the
 * activation buffers for max_n candidates. weights_host may be host memory or this
 * device's memory (read through unified addressing; the caller keeps it). *out is NULL
 * on failure. The denoiser is the black-box f_theta of §3 (a DiT); the block follows
 * Eq. 7. */
fb_status fb_init_model(const fb_cfg* cfg, const float* weights_host, fb_model** out);
/* fb_free: waits for the model's stream and its offload copies, then releases what the
 * model owns (device memory, its own streams, events, the pinned error word). NULL is
 * allowed. A stream given with fb_set_stream stays the caller's. */
void fb_free(fb_model* m);
/* stream: a cudaStream_t (NULL = the model's own stream). */
fb_status fb_set_stream(fb_model* m, void* stream);
/* fb_set_sm_budget: the number of SMs the model's launches may occupy (0 = all of the
 * device's). Persistent GEMM grids, the stream-K co-residency rule and the attention
 * kernel's CTA size are sized to it. Set it to the SM count of a partition whose stream
 * the model runs on (fb_sm_split_*): a GEMM that assumed more resident SM pairs than the
 * partition holds would leave its stream-K finishers waiting until their time limit.
 * FB_EINVAL outside [2, device SMs]. Waits for the model's stream first. */
fb_status fb_set_sm_budget(fb_model* m, int n_sms);

/* ---- SM partitions (an engineering entry point: the paper has no counterpart) ------
 * The paper runs generation and verification on separate GPUs (Sec. 5). On one GPU, the
 * draft pool (compute-bound, many waves) and the refinement of one candidate (a chain of
 * one-wave launches) can run side by side on disjoint SM sets. fb_sm_split_create splits
 * the current device's SMs into a group of n_sms (the driver may round the count to its
 * granularity) and the rest, each with a green context and a non-blocking stream in it;
 * kernels enqueued on a part's stream run only on that part's SMs, on the same device
 * memory. fb_sm_split_info(part 0 = the n_sms group, 1 = the rest) returns the part's
 * stream (a cudaStream_t; the split owns it) and its SM count, to pass to fb_set_stream
 * and fb_set_sm_budget. fb_sm_split_free waits for both streams and releases them; the
 * models that used them must be given other streams first. Errors: FB_EINVAL for n_sms
 * outside [2, device SMs - 2], FB_ECUDA when the driver offers no green contexts or a
 * call fails (nothing is left allocated). */
typedef struct fb_sm_split fb_sm_split;
fb_status fb_sm_split_create(int n_sms, fb_sm_split** out);
fb_status fb_sm_split_info(const fb_sm_split* split, int part, void** stream, int* sms);
void fb_sm_split_free(fb_sm_split* split);

/* fb_encode_text: text projection of the prompt embedding x (§3) and, per block, the
 * cross-attention keys and values; they do not change across steps or candidates and
 * are kept in the model. text_ctx: [text_len][text_dim] fp32, host or device. */
fb_status fb_encode_text(fb_model* m, const float* text_ctx);

/* ---- the draft and refine calls (§4.2 Stages 1 and 3) -------------------------
 * fb_draft: Stage 1 (Eq. 8) for n candidates (0 <= n <= max_n; n == 0 is a no-op).
 *  latents:  [n][latent_c][latent_h][latent_w] fp32, host or device; in: z_T per
 *            candidate; out: the latent after n_steps steps (the cached draft state).
 *  text_ctx: as fb_encode_text (encoded once per call).
 *  schedule: n_steps + 1 fp32 host values, strictly decreasing, in [0, 1]; step i goes
 *            from t = schedule[i] to t' = schedule[i+1] with the Euler update
 *            z <- z + (t' - t) v of the flow-matching ODE (App. A.1). Early stopping
 *            (§4.1, knob 1) is a schedule that ends before t = 0.
 *  skip_mask:  [n_steps][depth] uint8 host; 1 = skip the block (Eq. 6).
 *  proxy_plan: [n_steps][depth] int32 host; -1 = compute the block (Eq. 7); otherwise
 *            src_step | (order << 16), 0 <= order <= 2: the block's contribution
 *            Delta = B(h) - h is forecast by the Taylor expansion of Eqs. 3-5 from the
 *            contributions cached at the layer's most recent computed steps at or before
 *            src_step (most recent first; the order drops while fewer than order + 1
 *            exist) and added to h. The layer must have been computed at src_step,
 *            src_step < the current step, and the entry's skip bit must be 0.
 *            NULL skip_mask / proxy_plan mean "no skip" / "compute everything".
 *  Errors: FB_EINVAL (sizes, schedule), FB_EPLAN (plan rules above), FB_ENOMEM (proxy
 *  cache growth), FB_ECUDA. Argument and plan errors are reported before any work is
 *  enqueued and leave the latents unchanged; after FB_ECUDA a device buffer may be
 *  partly updated. */
fb_status fb_draft(fb_model* m, float* latents, int n, const float* text_ctx,
                   const float* schedule, int n_steps, const uint8_t* skip_mask,
                   const int32_t* proxy_plan);

/* fb_refine: Stage 3 (§4.2): resumes one latent [latent_c][latent_h][latent_w]
 * (host or device, in/out) with full computation (no skip, no proxy) over
 * full_schedule (n_steps + 1 values, as fb_draft). Valid because sampling is
 * Markovian: the result depends only on the latent it starts from. */
fb_status fb_refine(fb_model* m, float* latent, const float* text_ctx,
                    const float* full_schedule, int n_steps);

/* ---- sampler options: classifier-free guidance and the SDE step (App. A.1) -------
 * guidance / text_uncond: classifier-free guidance. When text_uncond is not NULL every
 * step also runs an unconditional pass (text_uncond, [text_len][text_dim] fp32, host or
 * device) through the same plan with its own proxy cache, and uses
 * v = v_u + guidance * (v_c - v_u). The conditional and unconditional rows form one
 * batch of 2n candidates, so 2n <= max_n is required (FB_EINVAL otherwise).
 * sde_a / noise: sde_a = 0 is the Euler step of the flow-matching ODE; sde_a > 0 is the
 * Euler-Maruyama step of the equivalent SDE (App. A.1):
 *   z <- z + [v + s^2/(2t) (z + (1-t) v)] dt + s sqrt(|dt|) eps,  dt = t' - t,
 *   s = sde_a sqrt(t / (1 - t)), evaluated at t' when t = 1,
 * with eps read from noise: [n_steps][n][latent_c][latent_h][latent_w] fp32 standard
 * normal draws supplied by the caller (host or device), required when sde_a > 0. */
typedef struct fb_sampler_opts {
  float guidance;
  const float* text_uncond;
  float sde_a;
  const float* noise;
  /* The cached state of Stage 3 (§4.2): per-layer activations kept with the latent so
   * that the refine can warm-start its activation proxies, read as each layer's contribution
   * Delta_l = B_l(h) - h from its last computed draft step (with that step's t):
   * keep_state (fb_draft_ex): != 0 keeps every candidate's state in the model after the
   *   call, for fb_state_offload (conditional rows under guidance);
   * state / warm_steps (fb_refine_ex): a state buffer of one candidate (fb_state_offload
   *   layout, host or device); the first warm_steps steps proxy every layer the state
   *   holds from it (order 0: h <- h + Delta_l), the other layers and steps compute.
   *   warm_steps = 0 or state = NULL is the plain refine. Not with guidance (FB_EINVAL). */
  int keep_state;
  const void* state;
  int warm_steps;
} fb_sampler_opts;

/* fb_draft_ex / fb_refine_ex: fb_draft / fb_refine with sampler options (opts may be
 * NULL: no guidance, ODE steps). fb_refine_ex's noise is [n_steps][1][C][H][W]. */
fb_status fb_draft_ex(fb_model* m, float* latents, int n, const float* text_ctx,
                      const float* schedule, int n_steps, const uint8_t* skip_mask,
                      const int32_t* proxy_plan, const fb_sampler_opts* opts);
fb_status fb_refine_ex(fb_model* m, float* latent, const float* text_ctx,
                       const float* full_schedule, int n_steps, const fb_sampler_opts* opts);

/* fb_pipeline_step: one step of a draft/refine pipeline in one call (§4.2 Stages 1 and
 * 3): refine_latent, the selected candidate of the previous pool, is refined with
 * `refiner` (as fb_refine_ex) on a worker thread while `drafter` drafts `latents` (as
 * fb_draft_ex) on the calling thread; the call returns when both are done. The two
 * models should run on the two parts of an fb_sm_split (fb_set_stream and
 * fb_set_sm_budget on each). refine_latent NULL: the draft alone (the first step).
 * The refine must not read `latents`: copy the selected candidate out before the next
 * step. Errors: FB_EINVAL for a NULL drafter, or a refine without a model of its own;
 * otherwise the draft's status if it failed, else the refine's, with its message
 * (prefixed "draft: " or "refine: ") in fb_last_error on the calling thread. */
fb_status fb_pipeline_step(fb_model* drafter, float* latents, int n, const float* text_ctx,
                           const float* draft_schedule, int n_draft_steps,
                           const uint8_t* skip_mask, const int32_t* proxy_plan,
                           const fb_sampler_opts* draft_opts, fb_model* refiner,
                           float* refine_latent, const float* refine_schedule,
                           int n_refine_steps, const fb_sampler_opts* refine_opts);

/* ---- cached-state offload (§4.2 Stage 3) --------------------------------------------
 * The paper moves the cached tensors to host memory during drafting and brings only the
 * selected candidate back for refinement; the copies are part of the wall-clock.
 * State layout of one candidate (fb_state_bytes bytes): depth fp32 values t_l (NaN: the
 * layer was never computed, no Delta), zero padding to byte 256, then depth blocks of
 * bf16 Delta_l [tokens][dim] (zeros where t_l is NaN).
 * fb_state_offload copies the states of candidates first .. first + count - 1 of the last
 * fb_draft_ex call with keep_state to dst[0] .. dst[count - 1] (host or device, each
 * fb_state_bytes bytes) on a model-owned copy stream and returns at once; with pinned
 * host memory the copies overlap whatever the model runs next. They are issued layer by
 * layer (every candidate's layer 0, then layer 1, ...): a later call that rewrites the
 * cached contributions waits, per cache slot, only for the copies still reading it.
 * A buffer is complete only after fb_state_wait, which blocks until every issued copy
 * has finished. Errors: FB_ESTATE when the last draft did not keep its state (or a later
 * call reused the cache), FB_EINVAL for a bad range or a NULL pointer. */
fb_status fb_state_bytes(const fb_model* m, size_t* bytes);
fb_status fb_state_offload(fb_model* m, int first, int count, void* const* dst);
fb_status fb_state_wait(fb_model* m);

/* fb_plan_from_phi: expands phi = (S', n_skip, l_start, l_end, f_full) (§4.1,
 * "Configuration Space") into skip_mask [S'][depth] and proxy_plan [S'][depth]
 * (caller-allocated host arrays). Layers l_start..l_end are 1-indexed as in the paper
 * and are skipped at draft steps k >= n_skip; step k is a full step iff
 * k mod f_full == 0; on other steps every non-skipped layer is proxied with the given
 * order from the last full step. FB_EINVAL if 1 <= S' <= S, 1 <= l_start <= l_end <=
 * depth, f_full >= 1, n_skip >= 0, 0 <= order <= 2 do not all hold. */
fb_status fb_plan_from_phi(int S, int S_prime, int n_skip, int l_start, int l_end,
                           int f_full, int order, int depth, uint8_t* skip_mask,
                           int32_t* proxy_plan);

/* ---- Stage 2 selection (§4.2), host only ---------------------------------------
 * fb_select_elo: multi-stage selection over M drafts. scores: [M] pointwise verifier
 * scores (1..10), seeding Elo ratings r = 1500 + (s - 5) * 100. Keeps the top
 * ceil(rho1 M) by rating (ties: lower index), runs ceil(kappa M1) comparisons between
 * adjacent entries of the survivors sorted by rating (passes from the top, re-sorted
 * before each pass), keeps the top ceil(rho2 M1), plays every pair of those in rating
 * order, and writes the index with the highest rating to *winner. The paper gives
 * neither the base K nor the expected score: k_base (32 is usual) times 1.2 / 1.0 / 0.7
 * for the verifier's high / medium / low confidence, and E_a = 1 / (1 + 10^((r_b - r_a)
 * / 400)). compare(user, a, b, &confidence) returns non-zero if a is preferred and sets
 * confidence to 0 (high), 1 (medium) or 2 (low). out_ratings: [M] final ratings or NULL;
 * out_calls: number of pairwise calls or NULL. FB_EINVAL for bad arguments or a
 * confidence outside 0..2 (then treated as medium). Runs on the calling thread. */
typedef int (*fb_pair_verifier)(void* user, int a, int b, int* confidence);
fb_status fb_select_elo(const int32_t* scores, int M, double rho1, double rho2,
                        double kappa, double k_base, fb_pair_verifier compare, void* user,
                        int* winner, double* out_ratings, int* out_calls);

/* fb_block_forward: one block B_layer (Eq. 7) in place on h [n * tokens][dim] fp32
 * DEVICE memory (candidate-major rows), with the modulation of timestep t and the
 * text context of the last fb_encode_text (FB_ESTATE without one). */
fb_status fb_block_forward(fb_model* m, int layer, float* h, int n, float t);

/* fb_last_error: the message of the calling thread's last failed call (each thread has
 * its own; the string stays valid until that thread's next failing call). */
const char* fb_last_error(void);

/* ---- statistics ----------------------------------------------------------------
 * Per kernel class: launches, summed device time (ms; measured with CUDA events on the
 * model's stream while timing is on) and algorithmic FLOPs and bytes of the launches. */
enum {
  FB_K_GEMM_TC = 0,   /* tcgen05/TMEM GEMM (all epilogues) */
  FB_K_GEMM_SIMT,     /* CUDA-core GEMM for shapes the tcgen05 kernel does not tile */
  FB_K_ATTN_SELF,     /* self-attention */
  FB_K_ATTN_CROSS,    /* cross-attention */
  FB_K_NORM,          /* LayerNorm + modulation */
  FB_K_QKNORM,        /* q/k RMSNorm + RoPE */
  FB_K_PROXY,         /* activation-proxy residual add */
  FB_K_EMBED,         /* patch embedding */
  FB_K_HEAD,          /* head + Euler update */
  FB_K_SMALL,         /* timestep embedding, modulation, conversions */
  FB_K_COUNT
};
typedef struct fb_kstat {
  uint64_t launches;
  double ms, flops, bytes;
} fb_kstat;
/* fb_set_timing: `on` is a bit mask; bit k records CUDA events around every launch of
 * class k (FB_K_*), 0 stops timing. fb_get_stats waits for the model's stream and
 * copies the FB_K_COUNT counters (launch counts and algorithmic work are always kept,
 * times only for timed classes); fb_reset_stats zeroes them; fb_kernel_name gives a
 * class's name ("?" outside [0, FB_K_COUNT)). FB_EINVAL for a NULL model or output. */
fb_status fb_set_timing(fb_model* m, int on);
fb_status fb_get_stats(fb_model* m, fb_kstat* out /* [FB_K_COUNT] */);
fb_status fb_reset_stats(fb_model* m);
const char* fb_kernel_name(int kind);

/* ---- single-op entry points (DEVICE pointers; enqueued on the model's stream) ---
 * They run one kernel of the path on caller buffers, for kernel-level parity tests.
 *
 * fb_op_gemm: D[M][N] = A[M][K] * W[N][K]^T + bias[N] with epilogue `epi`:
 *   0: out bf16 = acc + bias
 *   1: out bf16 = gelu_tanh(acc + bias)
 *   2: out fp32 = resid[M][N] + gate[N] * (acc + bias)  (gate may be NULL = 1; resid may
 *      equal out, or be NULL = 0: out fp32 = gate * (acc + bias))
 *   3: as 2, and also delta bf16 = out - base[M][N] (fp32), base may equal out
 * A, W bf16 row-major, leading dimensions K; out / resid / base / delta leading
 * dimension N. impl: 0 = automatic (tcgen05 when N % 128 == 0 and K % 64 == 0: the
 * 2-SM cta_group::2 kernel when N % 256 == 0, else the 1-SM kernel), 1 = force the
 * CUDA-core kernel, 2 = force the 1-SM tcgen05 kernel (same shape rules), 3 = the 2-SM
 * kernel over whole 256 x 256 tiles only, 4 = the 2-SM kernel with the stream-K split:
 * every SM pair takes an equal share of the (tile, 64-wide K block) units and tiles cut
 * between pairs are summed from fp32 partials in the model's workspace, in K order (so
 * the result does not depend on timing). impl 4 needs N % 256 == 0 and at least 4 K
 * blocks per SM pair (ceil(M / 256) * N / 256 * K / 64 >= 4 * pairs), else FB_ECUDA;
 * impl 0 takes the stream-K split only when K >= 96 * 64 and the whole 256 x 256 tiles
 * number fewer than the SM pairs that can be resident (e.g. 1560 x 1536 x 8960), whole
 * tiles otherwise. */
/* fb_set_op_repeat: fb_op_gemm / fb_op_attention launch their kernel n >= 1 times back
 * to back (default 1), for timing a kernel without a stream synchronisation per launch. */
fb_status fb_set_op_repeat(fb_model* m, int n);
fb_status fb_op_gemm(fb_model* m, int M, int N, int K, const void* A, const void* W,
                     const float* bias, int epi, void* out, const float* resid,
                     const float* gate, const float* base, void* delta, int impl);
/* fb_op_attention: O = softmax(Q K^T / sqrt(head_dim)) V per (batch, head), bf16 row
 * major; Q rows b*Lq..b*Lq+Lq-1 with row stride ldq elements, head h at column
 * h*head_dim; likewise K, V (kv_batch_rows = 0 shares one K/V across the batch,
 * otherwise the row offset between batches); O row stride ldo. impl: 0 = automatic
 * (the tcgen05 kernel for head_dim 128, the mma.sync kernel for 64), 1 = force the
 * mma.sync kernel, 2 / 3 = force the tcgen05 kernel with 128- / 256-query CTAs, 4 = force
 * the persistent 256-query kernel (at most one CTA per SM looping over the (batch, head,
 * query-tile pair) items; the automatic choice unless the 256-query form saves no
 * waves: both forms fit one wave, or Lq <= 128)
 * (2-4: head_dim 128 only, else FB_EINVAL). */
fb_status fb_op_attention(fb_model* m, const void* Q, int ldq, const void* K, int ldk,
                          const void* V, int ldv, void* O, int ldo, int batch, int Lq,
                          int Lkv, int kv_batch_rows, int heads, int head_dim, int impl);

/* ---- allocation-free stream-K GEMM (an engineering entry point: the paper has no
 * counterpart; it computes what fb_op_gemm with impl 4 computes) ---------------------
 * fb_gemm_streamk_noalloc: the same D = epi(A W^T + bias) as fb_op_gemm (same epi codes,
 * argument meaning and DEVICE-pointer layouts) with the stream-K split of the 2-SM
 * kernel, but with no model and no allocation of any kind: the partial accumulators,
 * the per-tile counters and the device error word live in static device arrays of the
 * library, sized for at most FB_NOALLOC_MAX_PAIRS SM pairs (76, a full GB300: 39.8 MB of
 * fp32 partials, 76 x 16 counters). Their addresses are looked up once per device on the
 * first call (cudaGetSymbolAddress, checked). The work is enqueued on `stream` (a
 * cudaStream_t; NULL = the legacy default stream) and the call waits for it, then reads
 * the error word.
 * State: the counters must be zero when a call starts; they are zero at load, every
 * successful call leaves them zero, and a call that reports a device error clears
 * them before returning. The error word is cleared at the start of every call. Calls
 * that overlap in time (other host threads, other streams) share these arrays and race:
 * serialise them.
 * SMs: the grid and the 4-blocks-per-pair rule use the whole device's SM count, and the
 * split relies on all of the device's SM pairs being resident at once. Do not pass a
 * stream of an SM partition (fb_sm_split): there completion depends on the order in
 * which the hardware starts clusters; a finisher of a cut tile whose contributors cannot
 * start until it leaves waits until the device wait limit (2 s by default) and the call
 * returns FB_ECUDA.
 * Errors: FB_EINVAL for a NULL pointer, a bad epi, N % 256 != 0, shapes the tcgen05
 * kernel does not take (K % 64, alignment), fewer than 4 K blocks per SM pair
 * (ceil(M / 256) * N / 256 * K / 64 < 4 * pairs) or a device with more than
 * FB_NOALLOC_MAX_PAIRS pairs; FB_ECUDA for a CUDA error or a device wait timeout. */
#define FB_NOALLOC_MAX_PAIRS 76
fb_status fb_gemm_streamk_noalloc(void* stream, int M, int N, int K, const void* A,
                                  const void* W, const float* bias, int epi, void* out,
                                  const float* resid, const float* gate, const float* base,
                                  void* delta);

/* ---- testing hooks (engineering entry points; the paper has no counterpart) ---------
 * fb_set_device_wait_limit: every device-side wait of the library's kernels (mbarrier
 * phases, stream-K counters) gives up after this many nanoseconds, records
 * "device wait timed out" in the call's error word, lets its copies in flight land,
 * frees its TMEM and returns; the call then returns FB_ECUDA and leaves the model
 * usable. ns = 0 restores the default (2 s). Applies to the current device and to every
 * model and call on it; tests shorten it to make a wait run out quickly. Not for use
 * while kernels of the library are running.
 * fb_test_fail_alloc: host-side failure injection for device allocations. After the call
 * the library counts its device allocations (every cudaMalloc it makes) from 0; the one
 * numbered k fails as an out-of-memory cudaMalloc would (the caller sees FB_ENOMEM).
 * k < 0 disarms. fb_test_alloc_calls: allocations counted since the last
 * fb_test_fail_alloc. Process-wide; not thread-safe against concurrent model creation.
 * fb_test_poison_counters: sets the model's stream-K tile counters (m = NULL: those of
 * fb_gemm_streamk_noalloc) to a large negative value, as a crashed launch could leave
 * them, so that the next stream-K finisher waits for a count no launch will reach. The
 * wait runs out at the device wait limit, the call returns FB_ECUDA and clears the
 * counters; the call after it computes normally. */
/* fb_probe_mma_rate: the tensor pipe's sustained rate on the current device, in MACs per SM
 * clock: every SM times (clock64) `reps` tcgen05.mma kind::f16 instructions of M = 128,
 * K = 16 and width n (64, 128 or 256) issued by each of `issuers` warps (1-4,
 * issuers * n <= 512 TMEM columns) into accumulators of their own; *mac_per_clk is
 * computed from the slowest SM. Allocates and
 * frees two small device buffers and synchronises the device. FB_EINVAL for arguments
 * outside those ranges, FB_ECUDA on a CUDA error. */
fb_status fb_probe_mma_rate(int issuers, int n, int reps, double* mac_per_clk);
/* fb_probe_mma_gap: the same rate (MACs per SM clock, slowest SM) when one thread per SM
 * issues 2048 batches of 8 instructions (M = N = 128, K = 16) and spins `gap` clocks
 * (0 .. 100000) after each batch: how much work the tensor pipe holds queued while its
 * issuing thread does something else. FB_EINVAL / FB_ECUDA as above. */
fb_status fb_probe_mma_gap(int gap, double* mac_per_clk);
/* fb_probe_mufu: results per SM clock (slowest SM) of one special-function operation,
 * op 0 = ex2.approx.ftz.f32, 1 = tanh.approx.f32, 2 = rcp.approx.ftz.f32, 3 =
 * ex2.approx.f16x2 (two results per instruction), with 256 threads per SM each running
 * 16 independent chains. FB_EINVAL / FB_ECUDA. */
fb_status fb_probe_mufu(int op, double* per_clk);
/* fb_probe_tmem_load: mean SM clocks from issuing four tcgen05.ld 32x32b.x32 (128 TMEM
 * columns of a warp's lane quarter) to the end of their wait, over 2000 repetitions by
 * 4 warps per SM, with the tensor pipe idle (busy = 0) or running M = N = 128 MMAs into
 * other columns (busy != 0). FB_EINVAL / FB_ECUDA. */
fb_status fb_probe_tmem_load(int busy, double* clocks);
/* fb_probe_mma_mix: MACs per SM clock (slowest SM) of 1024 batches shaped like one
 * attention step of one 128-query tile, issued by one thread per SM: 8 instructions
 * (M = N = 128, K = 16) into one accumulator, in form 0 (A and B K-major in shared
 * memory), 1 (B MN-major in shared memory, as V is read) or 2 (B MN-major, A read from
 * TMEM, as P is read), then 8 K-major shared-memory instructions into another. Warps
 * 1..loaders (0-7) meanwhile load 128 TMEM columns of their lane quarter, store 64 and
 * spin loader_gap clocks (0 .. 100000), as softmax warps do. Forms 3 and 4 issue one whole
 * attention step per batch instead (32 instructions: PV and S of two query tiles over
 * distinct operand slices, each descriptor built from its address), form 4 with the
 * attention's tcgen05.commit instructions; forms 5 and 6 are forms 3 and 4 with the
 * descriptors' lower words hoisted (one add per operand and instruction). Forms 7-13 are
 * forms 0-6 with the loaders also doing a softmax row's arithmetic (maximum, 128
 * exponentials, sum, bf16 packing) between load and store. FB_EINVAL / FB_ECUDA. */
fb_status fb_probe_mma_mix(int form, int loaders, int loader_gap, double* mac_per_clk);
fb_status fb_set_device_wait_limit(unsigned long long ns);
fb_status fb_test_fail_alloc(long k);
long fb_test_alloc_calls(void);
fb_status fb_test_poison_counters(fb_model* m);

#ifdef __cplusplus
}
#endif
#endif /* FLASHBON_H */
