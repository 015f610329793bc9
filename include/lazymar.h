/*
 * lazymar.h - C ABI of a GB300 (sm_103a) implementation of LazyMAR's cached
 * MAR decoding step (Yan et al., "LazyMAR: Accelerating Masked Autoregressive
 * Models via Feature Caching", ICCV 2025).
 *
 * A masked autoregressive (MAR) transformer is run once per decoding step over
 * a sequence of T = n_buffer + n_img tokens per image: n_buffer conditional
 * (class) tokens followed by the image tokens (Eq. 6; 64 + 256 tokens in the
 * paper's setting, Sec. 4.1). Bidirectional attention (Eq. 3) rules out a KV
 * cache, so LazyMAR caches features instead:
 *   - token cache (Sec. 3.2.1): after the first `sel_layers` blocks, each
 *     token's value matrix is compared with its value at the previous step
 *     (cosine similarity, Eq. 8); only the N least similar tokens are run
 *     through the remaining blocks (Eq. 9), attending over cached keys/values
 *     of the other tokens, and the results are written back into the cache;
 *   - condition cache (Sec. 3.2.2, Eq. 10): the difference between the
 *     conditional and unconditional outputs is stored on steps that run both
 *     classifier-free-guidance pathways and reused on steps that run only the
 *     conditional one;
 *   - periodic refresh (Sec. 1, Fig. 3): full steps recompute everything and
 *     refill both caches.
 *
 * Conventions for every entry point
 *   - Row layout: a batch of B cond/uncond pairs runs as rows 0..B-1
 *     (conditional pathway of pairs 0..B-1) and B..2B-1 (unconditional pathway
 *     of the same pairs). Feature tensors are row-major [rows, tokens, width].
 *   - dtype: LAZYMAR_BF16 tensors hold raw bfloat16 (uint16 storage),
 *     LAZYMAR_F32 tensors IEEE float32. Arithmetic accumulates in fp32 (fp64
 *     for the similarity of Eq. 8).
 *   - Pointers: unless stated otherwise a tensor pointer may be device memory or
 *     host memory (pinned or pageable). Host buffers are staged through
 *     library-owned device buffers on `stream`. In the step calls, inputs
 *     the device can address (device memory, page-locked host memory mapped
 *     under unified addressing) are gathered into the staging buffers by one
 *     copy kernel, pageable ones by cudaMemcpyAsync; the guided output is
 *     written by the CFG kernel straight into device memory or mapped
 *     page-locked host memory when it starts on a 16-byte boundary, and
 *     otherwise staged and copied out.
 *   - stream: a cudaStream_t (NULL = legacy default stream). Calls enqueue work
 *     and return without waiting; buffers must stay valid until the stream work
 *     has completed. Argument errors are returned immediately and enqueue
 *     nothing. Errors detected on the device (bounded waits that expired,
 *     out-of-range indices or labels) are latched in a device error word and
 *     reported by lazymar_sync / lazymar_device_check.
 *   - No call allocates device memory except lazymar_create and
 *     lazymar_select_tokens (stream-ordered scratch for the similarities).
 *   - A handle is not thread-safe; distinct handles are independent.
 */
#ifndef LAZYMAR_H
#define LAZYMAR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum lazymar_status {
  LAZYMAR_OK = 0,
  LAZYMAR_ERR_INVALID_ARG = 1,  /* bad pointer, size or enum value */
  LAZYMAR_ERR_OOM = 2,          /* device allocation failed */
  LAZYMAR_ERR_CUDA = 3,         /* a CUDA runtime call or launch failed */
  LAZYMAR_ERR_STATE = 4,        /* cached step before any full step, or batch changed */
  LAZYMAR_ERR_TIMEOUT = 5,      /* a bounded device-side wait expired */
  LAZYMAR_ERR_UNSUPPORTED = 6,  /* shape outside what the kernels support */
  LAZYMAR_ERR_DEVICE = 7        /* a kernel found a bad index or label on the device */
} lazymar_status;

typedef enum lazymar_dtype { LAZYMAR_F32 = 0, LAZYMAR_BF16 = 1, LAZYMAR_E4M3 = 2 } lazymar_dtype;

/* Which representation of block sel_layers-1 the similarity of Eq. 8 compares:
 * the attention value matrix (Sec. 4.4 "value matrix instead of features";
 * default) or the block's output features (Eq. 8 as printed). */
typedef enum lazymar_criterion {
  LAZYMAR_CRITERION_VALUE = 0,
  LAZYMAR_CRITERION_FEATURE = 1
} lazymar_criterion;

/* Which tokens fill the recompute budget N of a cached step (Sec. 4.4,
 * Table 3 "token selection strategies"). LEAST_SIMILAR: the N tokens least
 * similar to their cached values (strategy V, LazyMAR's default; recompute
 * least similar = cache most similar). MOST_SIMILAR: the N most similar
 * (strategy IV: cache the minimum-similarity tokens). RANDOM: the N tokens
 * with the smallest caller-drawn 32-bit keys (strategy III; the random draw is
 * an input). Ties go to the lower token index; a NaN similarity counts as
 * -inf. An optional per-token priority class (uint8, higher first) is applied
 * before the rule: it expresses the strategies that choose by token type, for
 * example the observation-based strategy of Sec. 3.2.1 (priority 1 for tokens
 * decoded at steps t-1 and t) or strategies I/II (priority 1 for decoded,
 * respectively still-masked, tokens). */
typedef enum lazymar_select_rule {
  LAZYMAR_SELECT_LEAST_SIMILAR = 0,
  LAZYMAR_SELECT_MOST_SIMILAR = 1,
  LAZYMAR_SELECT_RANDOM = 2
} lazymar_select_rule;

/* Model and capacity. width % 128 == 0, head width (width/heads) 64 or 80 for
 * bf16 (any divisor of width up to 128 for f32), token_dim <= 64,
 * 1 <= sel_layers <= depth, 1 <= max_batch (pairs). */
typedef struct lazymar_config {
  int depth;       /* transformer blocks L (encoder + decoder stacked) */
  int width;       /* D */
  int heads;       /* H */
  int mlp_ratio;   /* MLP hidden = mlp_ratio * D */
  int n_buffer;    /* conditional (class) tokens C of Eq. 6 */
  int n_img;       /* image tokens */
  int token_dim;   /* latent width of an image token (16 for KL-16) */
  int n_classes;   /* rows of the class-embedding table */
  int max_batch;   /* largest B (pairs) any step will use */
  int sel_layers;  /* s: blocks always run in full; Eq. 8 compares block s-1 */
  int dtype;       /* lazymar_dtype of weights, activations and caches */
  int criterion;   /* lazymar_criterion */
  float ln_eps;    /* LayerNorm epsilon */
  int select_rule; /* lazymar_select_rule of the cached steps (0 = strategy V) */
  int qkv_e4m3;    /* 1: the Q/K/V projection of blocks s..L-1 on the recomputed
                    * tokens runs on 8-bit tensor cores: LN1 output rounded to
                    * E4M3 (unit scale), W_qkv rounded to E4M3 with one scale
                    * per output channel (max |w| / 448), fp32 accumulation.
                    * bf16 only, width % 128 == 0. The paper ran FP16; this is
                    * an extension, within the bf16 parity tolerance on every
                    * configuration (E4M3 in the other GEMMs is not: see the
                    * design notes). 0: bf16 throughout. */
} lazymar_config;

/* Weights of one pre-LN block, fp32, [out, in] layout (y = x W^T + b).
 * Read once by lazymar_create (host or device pointers) and converted to the
 * configured dtype (bf16: round to nearest even). */
typedef struct lazymar_block_weights {
  const float *ln1_g, *ln1_b;  /* [D] */
  const float *w_qkv, *b_qkv;  /* [3D, D], [3D]; rows 0..D-1 Q, D..2D-1 K, 2D..3D-1 V */
  const float *w_o, *b_o;      /* [D, D], [D] */
  const float *ln2_g, *ln2_b;  /* [D] */
  const float *w1, *b1;        /* [mlp_ratio*D, D], [mlp_ratio*D] */
  const float *w2, *b2;        /* [D, mlp_ratio*D], [D] */
} lazymar_block_weights;

typedef struct lazymar_weights {
  const float *pos_emb;    /* [T, D] position embedding, added at every position */
  const float *class_emb;  /* [n_classes, D]; buffer tokens of the cond pathway */
  const float *mask_emb;   /* [D]; masked image tokens */
  const float *embed_w;    /* [D, token_dim]; decoded image tokens */
  const float *embed_b;    /* [D] */
  const float *lnf_g, *lnf_b;            /* [D] final LayerNorm */
  const lazymar_block_weights *blocks;   /* host array of `depth` entries */
} lazymar_weights;

/* Inputs of one decoding step for B pairs (both pathways share them). The two
 * selection inputs are read by cached steps only, for the rows that step runs
 * (2B, or B when it reuses the condition cache), and may be NULL (RANDOM
 * requires select_keys). */
typedef struct lazymar_step_in {
  const float *latents;   /* [B, n_img, token_dim] fp32; ignored where masked */
  const uint8_t *mask;    /* [B, n_img], 1 = still masked, 0 = decoded */
  const int32_t *labels;  /* [B] class labels in [0, n_classes) */
  int batch;              /* B, 1 <= B <= max_batch */
  const uint8_t *select_priority; /* [rows, T] priority classes, higher recomputed first */
  const uint32_t *select_keys;    /* [rows, T] random keys of LAZYMAR_SELECT_RANDOM */
} lazymar_step_in;

typedef struct lazymar_handle lazymar_handle;

/* Creates a model instance on the current CUDA device: copies and converts the
 * weights and allocates the token cache (keys/values of blocks s..L-1), the
 * selection reference, the output cache, the condition cache and all scratch
 * for max_batch pairs. The handle owns all of it until lazymar_destroy.
 * Returns INVALID_ARG / UNSUPPORTED for bad configurations, OOM if the device
 * allocation fails. */
lazymar_status lazymar_create(const lazymar_config *cfg, const lazymar_weights *w,
                              lazymar_handle **out);
void lazymar_destroy(lazymar_handle *h);

/* Full (refresh) step, Fig. 3 and Sec. 1 "periodic cache-reuse-refreshment":
 * every block over every token of both pathways (2B rows); refills the token
 * cache (C_token^l := F^l(X), Sec. 3.2.1), the selection reference and the
 * condition cache (Eq. 10).
 *   z_out      [2B, n_img, D] final features of the image tokens (may be NULL)
 *   guided_out [B, n_img, D]  u + gamma (c - u) (may be NULL) */
lazymar_status lazymar_full_step(lazymar_handle *h, const lazymar_step_in *in, float gamma,
                                 void *z_out, void *guided_out, void *stream);

/* Cached step (Sec. 3.2, Eq. 8-10). Blocks 0..s-1 run over all tokens; at
 * block s-1 Eq. 8 picks, per row, the n_compute tokens whose value matrix is
 * least similar to the previous step's (ties to the lower token index) and the
 * selection reference is overwritten; blocks s..L-1 run only those tokens
 * (their queries attend over all T keys, cached for the others, Eq. 9) and
 * write their keys, values and output features back into the cache.
 *   n_compute       N, 0 <= N <= T tokens recomputed per row
 *   use_cond_cache  1: run only the conditional rows (B) and rebuild the
 *                   unconditional output as c - delta (Sec. 3.2.2);
 *                   0: run both pathways (2B rows) and refresh delta
 *   idx_in          optional [rows, N] int32 caller-chosen I_compute (strictly
 *                   increasing per row, values in [0, T)); replaces Eq. 8's
 *                   choice (the selection reference is still updated)
 *   idx_out         optional [rows, N] int32: the I_compute used, ascending
 *   z_out, guided_out as for lazymar_full_step.
 * Returns STATE before the first full step or when B differs from it. */
lazymar_status lazymar_cached_step(lazymar_handle *h, const lazymar_step_in *in, int n_compute,
                                   int use_cond_cache, float gamma, const int32_t *idx_in,
                                   int32_t *idx_out, void *z_out, void *guided_out, void *stream);

/* Token selection of Eq. 8 on caller buffers (device pointers only).
 * v_cur, v_cache: [rows, T, D] in `dtype`. For every row: S_t = cosine of
 * v_cur[t] and v_cache[t] over D (fp64 accumulation of exact products,
 * S = dot / sqrt(max(|a|^2 |b|^2, 1e-16)), NaN counted as -inf); I_compute =
 * the n_compute smallest S, ties to the lower index, written ascending to
 * idx_out [rows, n_compute]. Then v_cache := v_cur. D % 8 == 0.
 * Allocates rows*T doubles of stream-ordered scratch (cudaMallocAsync). */
lazymar_status lazymar_select_tokens(int dtype, const void *v_cur, void *v_cache, int rows, int T,
                                     int D, int n_compute, int32_t *idx_out, void *stream);

/* lazymar_select_tokens under a selection rule (lazymar_select_rule, Table 3)
 * with optional per-token priority classes: tokens are taken by priority
 * descending, then the rule, then index ascending. priority [rows, T] uint8
 * may be NULL; keys [rows, T] uint32 are required for LAZYMAR_SELECT_RANDOM
 * and ignored otherwise. The similarities are computed and v_cache := v_cur
 * under every rule. Device pointers only; same scratch as
 * lazymar_select_tokens. */
lazymar_status lazymar_select_tokens_ex(int dtype, const void *v_cur, void *v_cache, int rows, int T,
                                        int D, int n_compute, int rule, const uint8_t *priority,
                                        const uint32_t *keys, int32_t *idx_out, void *stream);

/* lazymar_select_tokens without any device allocation. The paper has no
 * counterpart: this entry point exists for callers that may not allocate
 * device memory once running (a serving loop that fixes its memory budget at
 * start-up, a plug-in whose host framework owns the device allocator). Same
 * arguments, semantics and results as lazymar_select_tokens; device pointers
 * only. The similarity scratch is a fixed array inside the library, holding
 * LAZYMAR_SELECT_NOALLOC_MAX_TOKENS doubles (2 MiB) on every device that loads
 * it, until the process exits; rows * T above that limit returns
 * LAZYMAR_ERR_INVALID_ARG. Every call looks up the array's device address on
 * the current device (cudaGetSymbolAddress, which allocates nothing), so the
 * address stays right after a device reset; the first call on a device also
 * loads the library's device code there, so make it before any stream
 * capture. All calls
 * share the one array and leave their similarities in it: calls whose work
 * can overlap on the GPU (different streams, or different host threads) race
 * and must be serialised by the caller. No cudaMalloc, cudaFree or other
 * allocating call is made. */
#define LAZYMAR_SELECT_NOALLOC_MAX_TOKENS 262144
lazymar_status lazymar_select_tokens_noalloc(int dtype, const void *v_cur, void *v_cache, int rows,
                                             int T, int D, int n_compute, int32_t *idx_out,
                                             void *stream);

/* Classifier-free guidance with the condition cache (Eq. 7 read as
 * u + gamma (c - u), Eq. 10), elementwise over n elements (device pointers):
 *   mode 0 GUIDE:   guided = u + gamma (c - u)
 *   mode 1 REFRESH: delta := c - u; guided = u + gamma (c - u)
 *   mode 2 REUSE:   u' = c - delta; guided = u' + gamma (c - u');
 *                   z_uncond_out := u' (if not NULL). z_uncond is unused.
 * guided_out may be NULL. Arithmetic in fp32. */
enum { LAZYMAR_CFG_GUIDE = 0, LAZYMAR_CFG_REFRESH = 1, LAZYMAR_CFG_REUSE = 2 };
lazymar_status lazymar_cfg_combine(int dtype, int mode, const void *z_cond, const void *z_uncond,
                                   void *delta, float gamma, size_t n, void *z_uncond_out,
                                   void *guided_out, void *stream);

/* Component entry points: the kernels the steps run, on caller buffers
 * (device pointers only), for parity tests and for callers composing their
 * own pipeline. The kernels start while the previous kernel of the library on
 * the same stream finishes (programmatic dependent launch) and wait for it
 * before touching activations; weights (W of lazymar_linear, g and b of
 * lazymar_layernorm) are read before that wait, so they must not be outputs
 * of the library's kernel launched just before on the same stream. */

/* y = a W^T + bias with a fused epilogue, a [M, K], W [N, K] (row-major,
 * dtype), bias [N] (dtype, may be NULL). bf16 runs on the tcgen05 tensor cores
 * (K % 64 == 0, N % 128 == 0); f32 on CUDA cores (K % 4 == 0, N % 4 == 0).
 *   LAZYMAR_EPI_BIAS     out [M, ldo] dtype = y
 *   LAZYMAR_EPI_GELU     out [M, ldo] dtype = GELU(y) (erf form)
 *   LAZYMAR_EPI_RESIDUAL out [M, ldo] fp32 += y
 *   LAZYMAR_EPI_QKV      N = 3D: columns 0..D-1 -> out [M, D]; D..2D-1 ->
 *                        k_out[row_map[m], :]; 2D..3D-1 -> v_out[row_map[m], :]
 *                        (row_map NULL = identity; the cache scatter of Eq. 9)
 *   LAZYMAR_EPI_SILU     out [M, ldo] dtype = SiLU(y) = y sigmoid(y)
 * flags: 0 automatic tile width, 1 force 128, 2 force 256, 3 force 192, 4 force
 * 64 (bf16; a forced width of 192 or 256 that does not divide N falls back to
 * 128). */
enum { LAZYMAR_EPI_BIAS = 0, LAZYMAR_EPI_GELU = 1, LAZYMAR_EPI_RESIDUAL = 2, LAZYMAR_EPI_QKV = 3,
       LAZYMAR_EPI_SILU = 4 };
lazymar_status lazymar_linear(int dtype, int epilogue, const void *a, const void *w,
                              const void *bias, int M, int N, int K, void *out, int ldo,
                              void *k_out, void *v_out, const int32_t *row_map, int flags,
                              void *stream);

/* lazymar_linear with E4M3 operands (kind::f8f6f4 tensor cores, fp32
 * accumulation): a [M, K] and w [N, K] hold E4M3 bytes, wscale [N] fp32 the
 * per-output-column scale of w; y = (a w^T) * wscale + bias (bias bf16, may be
 * NULL). Epilogues BIAS, GELU (bf16 out) and QKV (bf16 Q/K/V, K/V scattered
 * through row_map) as for lazymar_linear. K % 128 == 0, N % 128 == 0. The
 * paper has no 8-bit arithmetic; this is the Q/K/V projection of a
 * configuration with qkv_e4m3 set. */
lazymar_status lazymar_linear_e4m3(int epilogue, const void *a, const void *w, const float *wscale,
                                   const void *bias, int M, int N, int K, void *out, int ldo, void *k_out,
                                   void *v_out, const int32_t *row_map, int flags, void *stream);

/* E4M3 copy of a bf16 weight matrix w [rows, cols] (cols % 8 == 0) with one
 * scale per row: scale[r] = max_c |w[r, c]| / 448 (1 for a zero row),
 * q[r, c] = E4M3(w[r, c] / scale[r]) (nearest, ties to even, saturating).
 * Device pointers: q [rows, cols] bytes, scale [rows] fp32. */
lazymar_status lazymar_quantize_e4m3(const void *w, int rows, int cols, void *q, float *scale, void *stream);

/* Multi-head bidirectional attention of Eq. 3 with a query subset: for each row
 * r and head h, O[r, j] = softmax(Q[r, j] K[r]^T / sqrt(dh)) V[r] over all T
 * keys. q, o: [rows, n_q, heads*head_dim]; k, v: [rows, T, heads*head_dim]
 * (dtype). bf16: head_dim 64 or 80, tcgen05 tensor cores with TMA-staged K/V. */
lazymar_status lazymar_attention(int dtype, const void *q, const void *k, const void *v, void *o,
                                 int rows, int n_q, int T, int heads, int head_dim, void *stream);

/* LayerNorm over D of fp32 rows: y[m] = LN(x[row_map ? row_map[m] : m]) * g + b,
 * y in dtype, g/b in dtype; dtype LAZYMAR_E4M3: g/b bf16, y E4M3 bytes (unit
 * scale, saturating at 448). D % 128 == 0, D <= 2048. */
lazymar_status lazymar_layernorm(int dtype, const float *x, const int32_t *row_map, const void *g,
                                 const void *b, void *y, int M, int D, float eps, void *stream);

/* Schedule of periodic cache-reuse-refreshment (host only, no GPU): steps
 * k < k0 are full, then full whenever (k - k0) % tau == 0; other steps are
 * cached and reuse the condition cache when use_cond_cache and tau_cfg > 0 and
 * (k - k0) % tau_cfg != 0. Returns bit 0 = full step, bit 1 = reuse the
 * condition cache, or -1 for invalid arguments. */
int lazymar_plan_step(int k, int k0, int tau, int tau_cfg, int use_cond_cache);

/* Copies the selection reference of the first `rows` rows, [rows, T, D] in the
 * handle's dtype, to dst (device or host memory, caller-owned), on `stream`.
 * The reference is C^{l=3} of Eq. 8: the representation each row had when it
 * last ran (after a cached step, this step's block s-1 value matrix or
 * features). Reading it before and after a cached step gives the two inputs
 * of that step's Eq. 8 selection. Returns STATE before the first full step,
 * INVALID_ARG for rows outside 1..2 max_batch or a NULL dst. */
lazymar_status lazymar_read_reference(lazymar_handle *h, int rows, void *dst, void *stream);

/* Step execution. Each step first copies its inputs (latents, mask, labels,
 * idx_in) into handle-owned buffers on `stream`, so the device work reads
 * fixed addresses. That work (embedding through the final LayerNorm) runs
 * eagerly the first time a (step kind, B, N, cond reuse, idx_in given)
 * combination is seen, is captured into a CUDA graph the second time (on a
 * stream of the handle's) and replayed on `stream` from then on; the CFG
 * combine and the output copies are launched after it, so gamma may change
 * from call to call. enable = 0 runs every step
 * eagerly. While profiling is on, each combination is captured on its first
 * use together with an event record around every launch, into a graph of its
 * own, and replayed; the per-kernel times are then device times, free of the
 * host's launch submission. */
lazymar_status lazymar_set_graphs(lazymar_handle *h, int enable);

/* Waits for `stream`, then reports (and clears) errors the handle's kernels
 * latched on the device: TIMEOUT, DEVICE, or CUDA for an asynchronous fault. */
lazymar_status lazymar_sync(lazymar_handle *h, void *stream);

/* As lazymar_sync for the component entry points of the current device. */
lazymar_status lazymar_device_check(void *stream);

/* Failure-detection self-test (no counterpart in the paper): launches one CTA
 * that waits on an mbarrier nothing completes, with a wait limit of limit_us
 * microseconds (1..1000000), the same bounded wait every pipelined kernel
 * uses. The wait runs out, the kernel raises LAZYMAR_ERR_TIMEOUT in the
 * component error word and returns; the next lazymar_device_check on the
 * stream reports LAZYMAR_ERR_TIMEOUT (and clears it), and the device stays
 * usable. Returns INVALID_ARG outside the limit range. */
lazymar_status lazymar_selftest_wait(int limit_us, void *stream);

/* ------------------------------------------------------------------------
 * Diffusion head (Sec. 4.1: each decoded token's continuous latent is drawn
 * by a per-token denoiser run for 100 diffusion steps of the standard sampler;
 * its features z come from the transformer's final LayerNorm, a7).
 *
 * Denoiser (per token row r with latent x, training step t, feature z):
 *   y = t_emb(t) + W_c z + b_c,  t_emb = Linear(SiLU(Linear(sinusoids(t))))
 *   h = W_in x + b_in
 *   per block: (shift, scale, gate) = W_ada SiLU(y) + b_ada
 *              h += gate * MLP(LN(h) (1 + scale) + shift),  MLP = Linear, SiLU, Linear
 *   (shift, scale) = W_fada SiLU(y) + b_fada
 *   out = W_out (LN(h) (1 + scale) + shift) + b_out = [eps, v]  (2 token_dim)
 * LN without gain or shift. Sampler: cosine schedule over n_train training
 * steps, n_steps kept steps round(i (n_train - 1) / (n_steps - 1)); per kept
 * step j = n_steps-1 .. 0 the network runs on (x, z_cond) and (x, z_uncond),
 * eps = eps_u + gamma (eps_c - eps_u), v from the conditional run, and
 *   x <- mean(x, eps) + [j > 0] exp(log_var(v) / 2) temperature noise
 * with the Gaussian posterior mean and the learned-range log variance
 * (frac = (v + 1) / 2 between log beta_j and the clipped log posterior
 * variance). Weights are fp32 (host or device), stored as bf16 at create;
 * the matrix products run on the tcgen05 tensor cores (width % 128 == 0,
 * cond_dim % 64 == 0, freq_dim % 128 == 0).
 * ------------------------------------------------------------------------ */
typedef struct lazymar_head lazymar_head;
typedef struct lazymar_head_config {
  int token_dim;   /* latent width (16 for KL-16), 1..64 */
  int cond_dim;    /* width of z (the transformer width) */
  int z_dtype;     /* LAZYMAR_BF16 or LAZYMAR_F32: dtype of the z buffers */
  int width;       /* denoiser width */
  int depth;       /* residual blocks */
  int freq_dim;    /* sinusoidal timestep features */
  int n_train;     /* training steps of the noise schedule (1000) */
  int n_steps;     /* sampling steps (100), 1..n_train */
  int max_tokens;  /* tokens per lazymar_head_sample call */
  float ln_eps;    /* LayerNorm epsilon (1e-6) */
} lazymar_head_config;
typedef struct lazymar_head_block_weights {
  const float *ada_w, *ada_b;  /* [3 width, width], [3 width]: shift, scale, gate rows */
  const float *w1, *b1;        /* [width, width], [width] */
  const float *w2, *b2;        /* [width, width], [width] */
} lazymar_head_block_weights;
typedef struct lazymar_head_weights {
  const float *t_w1, *t_b1;    /* [width, freq_dim], [width] */
  const float *t_w2, *t_b2;    /* [width, width], [width] */
  const float *c_w, *c_b;      /* [width, cond_dim], [width] */
  const float *in_w, *in_b;    /* [width, token_dim], [width] */
  const lazymar_head_block_weights *blocks;  /* depth entries */
  const float *f_ada_w, *f_ada_b;  /* [2 width, width], [2 width]: shift, scale rows */
  const float *out_w, *out_b;      /* [2 token_dim, width], [2 token_dim] */
} lazymar_head_weights;

/* Validates the configuration, copies the weights and precomputes the
 * schedule and the time embeddings of the kept steps on the current device. */
lazymar_status lazymar_head_create(const lazymar_head_config *cfg, const lazymar_head_weights *w,
                                   lazymar_head **out);
void lazymar_head_destroy(lazymar_head *hd);

/* Draws the latents of the tokens decoded at one decoding step.
 *   z      device [2B, n_img, cond_dim] (z_dtype): rows 0..B-1 the conditional
 *          features of pairs 0..B-1, rows B..2B-1 the unconditional ones (the
 *          z output of lazymar_full_step / lazymar_cached_step)
 *   pos    [B, n_new] image positions decoded now (host or device), each in
 *          0..n_img-1; token m = b n_new + k is pair b's position pos[b][k]
 *   noise  [n_steps, B n_new, token_dim] fp32 (host or device): noise[0] the
 *          starting latents, noise[i] the noise added after denoising step i
 *   x_out  [B n_new, token_dim] fp32 (host or device)
 * B n_new <= max_tokens. Asynchronous on `stream`; the sampling loop is
 * captured into a CUDA graph per token count and replayed. Positions out of
 * range raise LAZYMAR_ERR_DEVICE at the next check. */
lazymar_status lazymar_head_sample(lazymar_head *hd, const void *z, int B, int n_img, const int32_t *pos,
                                   int n_new, const float *noise, float gamma, float temperature,
                                   float *x_out, void *stream);
/* One guided network evaluation at kept step j (0 = last), for tests:
 * out [2 B n_new, 2 token_dim] fp32 (host or device) = the network output of
 * the conditional rows (0..M-1) and the unconditional rows (M..2M-1) for
 * latents x [B n_new, token_dim] fp32. */
lazymar_status lazymar_head_eval(lazymar_head *hd, const void *z, int B, int n_img, const int32_t *pos,
                                 int n_new, const float *x, int j, float *out, void *stream);
/* Kernel launches issued by this head so far (graph replays count their
 * kernels), and the same for algorithmic flops. */
lazymar_status lazymar_head_counters(lazymar_head *hd, long long *launches, double *flops);
/* Waits for the head's work on `stream` and reports device errors. */
lazymar_status lazymar_head_sync(lazymar_head *hd, void *stream);
/* The sampler's schedule as the head computes it (host only, no GPU): for
 * kept steps j = 0..n_steps-1 (j = 0 the last denoising step),
 * kept[j] = round(j (n_train - 1) / (n_steps - 1)) (ties to even), and
 * consts[4 j + 0..3] = 1 / sqrt(1 - beta_j), beta_j / (sqrt(1 - beta_j)
 * sqrt(1 - alpha_bar_j)), log beta_j and the clipped log posterior variance,
 * so that mean = consts[0] x - consts[1] eps. Either output may be NULL.
 * Returns INVALID_ARG unless 1 <= n_steps <= n_train. */
lazymar_status lazymar_head_schedule(int n_train, int n_steps, int32_t *kept, float *consts);

/* Per kernel class: kernel launches (a GEMM split into two launches counts
 * two), algorithmic flops and bytes, and (while profiling is on) device time
 * from CUDA events recorded around each call on its stream (timed_launches
 * counts those event pairs; one pair encloses both launches of a split GEMM).
 * lazymar_get_stats waits for the recorded events. */
enum {
  LAZYMAR_K_GEMM = 0, LAZYMAR_K_ATTENTION = 1, LAZYMAR_K_LAYERNORM = 2, LAZYMAR_K_SELECT = 3,
  LAZYMAR_K_EMBED = 4, LAZYMAR_K_CFG = 5, LAZYMAR_K_OTHER = 6, LAZYMAR_K_COUNT = 7
};
typedef struct lazymar_kernel_stats {
  long long launches;
  long long timed_launches;
  double ms;
  double flops;
  double bytes;
} lazymar_kernel_stats;
typedef struct lazymar_stats {
  lazymar_kernel_stats k[LAZYMAR_K_COUNT];
} lazymar_stats;
lazymar_status lazymar_set_profiling(lazymar_handle *h, int enable);
lazymar_status lazymar_get_stats(lazymar_handle *h, lazymar_stats *out);
lazymar_status lazymar_reset_stats(lazymar_handle *h);

const char *lazymar_status_string(lazymar_status s);
/* Text of the last error on the calling thread (empty if none). */
const char *lazymar_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* LAZYMAR_H */
