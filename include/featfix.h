/*
 * featfix.h -- C ABI of the GB300 (sm_103a) FeatFix cached-DiT denoising path.
 *
 * FeatFix ("Reuse What You Verify through Local Exact-Feature Correction for
 * Faster Cached Diffusion Inference") runs a cached diffusion-transformer
 * sampler in which every block l at every timestep t either emits a cheap
 * draft of its output (reuse or an order-K Taylor forecast, Eq. 2) or runs the
 * exact block B_l(u; t, c) (Eq. 1).  At full-refresh steps every block is
 * exact; at a fixed sparse set S of (timestep, layer) sites the draft and the
 * exact output are both formed from the same incoming state (Eq. 3), their
 * relative discrepancy is logged (Eq. 4) and the exact output is forwarded in
 * place of the draft (Eq. 5).  Section 3.3 defines the site set, the Verify
 * arm (forwards the draft, discards the exact output), the Exact-only arm
 * (forwards the exact output without forming the draft) and the accounting
 * of refreshes, paid checks and forwarded corrections.
 *
 * Conventions for every entry point:
 *  - Pointers named dev_* / "device" are CUDA device pointers on the device
 *    that was current when the context was created; *_host pointers are host
 *    memory.  The library never frees caller memory.
 *  - Every call returns a featfix_status and never aborts, traps or exits.
 *    Asynchronous device errors surface as FEATFIX_ERR_CUDA at the next
 *    synchronising call (featfix_get_log, featfix_sample_host).  The message
 *    of the last failure is featfix_last_error(ctx).
 *  - A context is not thread-safe; all of its device work is ordered on the
 *    CUDA stream given to featfix_create.
 *  - Indices are 0-based: steps 0..steps-1, layers 0..L-1 where L = n_dual +
 *    n_single (MMDiT) or n_dual (DiT; the DiT blocks are counted in n_dual).
 */
#ifndef FEATFIX_H
#define FEATFIX_H

#include <stddef.h>

#if defined(__GNUC__)
#define FEATFIX_API __attribute__((visibility("default")))
#else
#define FEATFIX_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum featfix_status {
  FEATFIX_OK = 0,
  FEATFIX_ERR_INVALID_ARG = 1,   /* null pointer, bad size or unsupported shape */
  FEATFIX_ERR_SCHEDULE = 2,      /* schedule rule violated (see featfix_set_schedule) */
  FEATFIX_ERR_STATE = 3,         /* call out of order (no schedule, step not next) */
  FEATFIX_ERR_OOM = 4,           /* device allocation failed */
  FEATFIX_ERR_CUDA = 5,          /* CUDA runtime / kernel error (incl. kernel watchdog) */
  FEATFIX_ERR_UNSUPPORTED = 6    /* valid request this build does not implement */
} featfix_status;

/* Arms of Section 3.3 plus the all-exact reference sampler. */
typedef enum featfix_mode {
  FEATFIX_MODE_FEATFIX = 0,      /* site: forward h_f, log d(h_d, h_f)          (Eq. 5) */
  FEATFIX_MODE_VERIFY = 1,       /* site: forward h_d, log d(h_d, h_f), drop h_f */
  FEATFIX_MODE_EXACT_ONLY = 2,   /* site: forward h_f, no draft, no log          */
  FEATFIX_MODE_VANILLA = 3       /* every block exact at every step, no cache    */
} featfix_mode;

enum { FEATFIX_ARCH_DIT = 0, FEATFIX_ARCH_MMDIT = 1 };
enum { FEATFIX_DTYPE_F32 = 0, FEATFIX_DTYPE_BF16 = 1 };
enum { FEATFIX_SAMPLER_EULER = 0, FEATFIX_SAMPLER_DDIM = 1 };
/* Plan entries (featfix_get_plan, featfix_plan_build). */
enum { FEATFIX_PLAN_EXACT = 0, FEATFIX_PLAN_DRAFT = 1, FEATFIX_PLAN_SITE = 2 };
/* featfix_set_schedule flags.  TAYLOR_RECURSIVE selects the recursive
 * finite-difference estimator of Eq. 2 (each order's difference divided by
 * the spacing of the two refreshes it joins) instead of the default
 * derivatives of the polynomial interpolating the last K+1 refreshes.  */
#define FEATFIX_FLAG_TAYLOR_RECURSIVE 1u
/* PER_BLOCK_DRAFT forces one draft kernel per block at every drafted step.
 * By default a drafted step without a FeatFix/Exact-only site is evaluated
 * in one pass: at a full-refresh step every block is exact and each block's
 * input is the previous block's output, so the per-block increments
 * telescope, sum_l R_l = x_L - x_0; the forecast of the whole step is then
 * x_0 + sum_j w_j (x_L - x_0)_{s_j}, the same value as chaining the L
 * per-block drafts (up to rounding).  A step with a FeatFix/Exact-only site
 * drafts each run of consecutive drafted blocks (before, between and after
 * its sites) in one pass: x + sum over the run's blocks of sum_j w_j R_j,
 * read and written once.  In the Verify arm every drafted step is evaluated
 * by the whole-step form (so its forwarded trajectory is the one without
 * sites) and the paid checks run on a shadow copy drafted run by run up to
 * the step's last site.  The flag restores one draft per block everywhere;
 * steps with a debug capture always run per block. */
#define FEATFIX_FLAG_PER_BLOCK_DRAFT 2u
/* SITE_UPDATES_HISTORY takes the other reading of where the finite
 * differences of Eq. 2 are estimated: a site's exact increment h^f - u
 * (Eq. 3) is pushed onto its block's history like a refresh, after the
 * site's own draft (and its discrepancy, Eq. 4) used the history before
 * it.  Later drafts of that block then interpolate its own refresh-and-site
 * steps (featfix_plan_build_blocks gives the per-block weights).  Default
 * off: sites leave the history alone, so the draft policy outside the site
 * set is the base policy's and Verify and FeatFix share their caches.
 * Drafted steps then run per block (no telescoping).                       */
#define FEATFIX_FLAG_SITE_UPDATES_HISTORY 4u
/* FUSED_LN fuses each adaLN LayerNorm-modulation of Eq. 1 that sits between
 * two dense layers into them (bf16 models, C a multiple of 64): the GEMM
 * that produces a block input (the embedding, the out-projection, fc2 /
 * linear2 of the previous block at a full-refresh or vanilla step) also
 * writes x (1 + scale) and per-row statistics of x, and the next layer
 * computes
 *   LN(x)(1 + scale)W^T + shift W^T
 *     = rstd [x (1 + scale)] W^T - rstd mean (1 + scale) W^T + shift W^T
 * with per-sample tables (1 + scale) W^T and shift W^T made once per
 * trajectory.  Blocks whose input is a draft (sites) and the final layer
 * keep the row kernel.  Same value up to rounding.  Off by default: the
 * extra epilogue work of the two GEMMs costs more than the row kernel it
 * removes (measured on GB300: DiT-XL/2 sampling 918 -> 677 steps/s,
 * HunyuanVideo 34.7 -> 31.3).                                              */
#define FEATFIX_FLAG_FUSED_LN 8u

/*
 * Model shape (Eq. 1's block B_l and the surrounding sampler).
 *  arch        FEATFIX_ARCH_DIT: class-conditional DiT, n_dual adaLN blocks.
 *              FEATFIX_ARCH_MMDIT: n_dual two-stream (text/image) blocks then
 *              n_single single-stream blocks, joint attention, rotary
 *              positions on image tokens.
 *  hidden=C, heads=H, head_dim=d (C == H*d, d % 8 == 0), mlp=M.
 *  in_ch/out_ch latent channels in / model output channels (out_ch >= in_ch;
 *              the first in_ch output channels drive the sampler).
 *  patch, patch_t  spatial / temporal patch (patch_t used when lat_f > 0).
 *  lat_f, lat_h, lat_w  latent frames (0 = image model), height, width.
 *  txt_tokens  N_txt (MMDiT), 0 for DiT.   n_classes  DiT label count; label
 *              n_classes is the null class.
 *  batch       B_lat samples; cfg != 0 doubles the model batch to
 *              B_model = 2*B_lat as [conditional ; unconditional] and guides
 *              with scale cfg_scale.
 *  rope_dims   0, 2 (row, col) or 3 (frame, row, col).
 *  dtype       FEATFIX_DTYPE_F32 or FEATFIX_DTYPE_BF16 (weights, residual
 *              stream and history; accumulation always fp32).
 *  sampler     FEATFIX_SAMPLER_EULER (flow matching, sigma_i = 1 - i/N) or
 *              FEATFIX_SAMPLER_DDIM (eta = 0, linear betas 1e-4..0.02 / 1000).
 */
typedef struct featfix_model_desc {
  int arch;
  int n_dual;
  int n_single;
  int hidden;
  int heads;
  int head_dim;
  int mlp;
  int in_ch;
  int out_ch;
  int patch;
  int patch_t;
  int lat_f;
  int lat_h;
  int lat_w;
  int txt_tokens;
  int n_classes;
  int batch;
  int cfg;
  float cfg_scale;
  int rope_dims;
  int dtype;
  int sampler;
} featfix_model_desc;

/* A paid verification site (Section 3.3): timestep `step`, block `layer`. */
typedef struct featfix_site {
  int step;
  int layer;
} featfix_site;

/* One logged paid check (Eq. 4 and its L2 analogue), epsilon = 1e-8. */
typedef struct featfix_site_log {
  int step;
  int layer;
  double rel_l1;     /* ||h_d - h_f||_1 / (||h_f||_1 + eps) */
  double rel_l2;     /* ||h_d - h_f||_2 / (||h_f||_2 + eps) */
  double norm_l1_f;  /* ||h_f||_1 */
  double norm_l2_f;  /* ||h_f||_2 */
} featfix_site_log;

/* Accounting of Section 3.3, for the current trajectory. */
typedef struct featfix_counters {
  int refresh_steps;  /* full-refresh timesteps executed (every step in vanilla) */
  int paid_checks;    /* sites executed (exact block paid at a skipped site)     */
  int forwarded;      /* exact outputs forwarded in place of the draft           */
  int steps_done;     /* denoising steps completed                                */
} featfix_counters;

typedef struct featfix_ctx featfix_ctx;

/* Number of weight tensors featfix_create expects for `desc` (-1 if the
 * description is invalid).  Order (nn.Linear convention, weight [out, in]):
 *  DiT   : t_fc1.w [C,256], t_fc1.b [C], t_fc2.w [C,C], t_fc2.b [C],
 *          y_emb [n_classes+1, C], x_emb.w [C, in_ch*P], x_emb.b [C],
 *          final.mod.w [2C,C], final.mod.b [2C], final.lin.w [P*out_ch, C],
 *          final.lin.b [P*out_ch], then per block l (10 tensors):
 *          mod.w [6C,C], mod.b [6C], qkv.w [3C,C], qkv.b [3C], proj.w [C,C],
 *          proj.b [C], fc1.w [M,C], fc1.b [M], fc2.w [C,M], fc2.b [C].
 *  MMDiT : t_fc1.w, t_fc1.b, t_fc2.w, t_fc2.b, img_in.w [C, in_ch*P],
 *          img_in.b, final.mod.w, final.mod.b, final.lin.w, final.lin.b, then
 *          per dual block (20): img_mod.w [6C,C], img_mod.b, txt_mod.w,
 *          txt_mod.b, img_qkv.w [3C,C], img_qkv.b, txt_qkv.w, txt_qkv.b,
 *          img_proj.w [C,C], img_proj.b, txt_proj.w, txt_proj.b,
 *          img_fc1.w [M,C], img_fc1.b, img_fc2.w [C,M], img_fc2.b,
 *          txt_fc1.w, txt_fc1.b, txt_fc2.w, txt_fc2.b; then per single block
 *          (6): mod.w [3C,C], mod.b, lin1.w [3C+M, C], lin1.b, lin2.w [C, C+M],
 *          lin2.b.
 *  P = patch*patch (* patch_t for video).  A patch feature is ordered
 *  (channel, frame offset, row offset, column offset); tokens are row-major
 *  over the patch grid.  Every tensor is contiguous in the model dtype.   */
FEATFIX_API int featfix_weight_count(const featfix_model_desc* desc);

/* Create a context for `desc` on the current CUDA device.
 *  dev_weights  array of featfix_weight_count(desc) device pointers in the
 *               order above (borrowed: must outlive the context).
 *  cuda_stream  a cudaStream_t (borrowed; NULL = legacy default stream).
 *  out          receives the context.
 * The context allocates its activation workspace (about 12*B_model*N*max(C,M)
 * elements) at creation and the refresh history when a schedule is set.
 * Errors: INVALID_ARG (bad desc, null pointer, misaligned weight: every
 * pointer must be 16-byte aligned), OOM, CUDA, UNSUPPORTED.                 */
FEATFIX_API featfix_status featfix_create(const featfix_model_desc* desc, const void* const* dev_weights,
                              int n_weights, void* cuda_stream, featfix_ctx** out);

/* Fix the schedule before sampling (Section 3.3: S is frozen before
 * evaluation and shared by all samples and by the Verify/FeatFix arms).
 *  steps          number of denoising steps N.
 *  refresh        the base policy's full-refresh steps (n_refresh entries).
 *  draft_order    K in Eq. 2 (0 = reuse), 0..3.
 *  sites          the site set S (n_sites entries, may be NULL if 0).
 *  mode           featfix_mode.   flags  FEATFIX_FLAG_*.
 * Rules (else FEATFIX_ERR_SCHEDULE): steps >= 1; step 0 is a refresh;
 * refresh steps distinct and in range; sites distinct, in range and not on a
 * refresh step; 0 <= K <= 3.  Allocates the history (K+1 increments per
 * block, dtype-sized) -- FEATFIX_ERR_OOM if it does not fit.  Resets the
 * trajectory.                                                               */
FEATFIX_API featfix_status featfix_set_schedule(featfix_ctx* ctx, int steps, const int* refresh, int n_refresh,
                                    int draft_order, const featfix_site* sites, int n_sites,
                                    int mode, unsigned flags);

/* One denoising step (Section 3: every block exact, drafted or a paid site
 * per the plan, then the final layer, guidance and the sampler update).
 *  dev_latent  float32 [B_lat, in_ch, (lat_f,) lat_h, lat_w], updated in place.
 *  step        must be 0 (starts a new trajectory) or the previous step + 1,
 *              else FEATFIX_ERR_STATE.
 *  dev_cond    DiT: int32 labels [B_model]; MMDiT: float32 text tokens
 *              [B_model, txt_tokens, C].  Under CFG the first B_lat rows are
 *              the conditional half, the rest the unconditional half.       */
FEATFIX_API featfix_status featfix_step(featfix_ctx* ctx, float* dev_latent, int step, const void* dev_cond);

/* A whole trajectory: x_T drawn from `seed` (SplitMix64 counters, word k =
 * mix(seed + (k+1)*0x9E3779B97F4A7C15), mapped to (0,1) as
 * ((w >> 11) + 0.5) * 2^-53, Box-Muller pairs (2m, 2m+1) -> elements 2m, 2m+1
 * of the flattened latent), then steps 0..steps-1.  `steps` must equal the
 * schedule's.  dev_latent_out receives x_0 (same layout as featfix_step).  */
FEATFIX_API featfix_status featfix_sample(featfix_ctx* ctx, unsigned long long seed, int steps,
                              const void* dev_cond, float* dev_latent_out);

/* featfix_sample with host buffers: copies cond_host to the device, samples,
 * copies x_0 back into latent_out_host and synchronises the stream.       */
FEATFIX_API featfix_status featfix_sample_host(featfix_ctx* ctx, unsigned long long seed, int steps,
                                   const void* cond_host, float* latent_out_host);

/* Logs of the current trajectory in execution order (synchronises the
 * stream).  Writes min(cap, available) entries into `out` (may be NULL when
 * cap == 0), the available count into *n and the counters (may be NULL).  */
FEATFIX_API featfix_status featfix_get_log(featfix_ctx* ctx, featfix_site_log* out, int cap, int* n,
                               featfix_counters* counters);

/* The plan of the current schedule: kinds [steps*L] (FEATFIX_PLAN_*),
 * k_eff [steps] (effective draft order, -1 where no draft is formed) and
 * the draft weights [steps*4] (weights of the 1..4 newest refresh
 * increments; unused entries 0).  Any output may be NULL.                   */
FEATFIX_API featfix_status featfix_get_plan(featfix_ctx* ctx, unsigned char* kinds, int* k_eff, double* weights);

/* Host-only plan builder (no context, no device): same rules and outputs as
 * featfix_set_schedule + featfix_get_plan for `n_layers` blocks.            */
FEATFIX_API featfix_status featfix_plan_build(int steps, int n_layers, const int* refresh, int n_refresh,
                                  int draft_order, const featfix_site* sites, int n_sites,
                                  int mode, unsigned flags, unsigned char* kinds, int* k_eff,
                                  double* weights);

/* Partial forwarding arms (the token- and channel-level alternatives to
 * whole-block forwarding the paper compares against, Section 3.2): at a
 * FeatFix site the forwarded output takes the exact block output h^f only
 * on the selected tokens or channels and the draft h^d elsewhere (the
 * discrepancy of Eq. 4 is still taken over the whole tensor).  The paper
 * does not say which tokens or channels are selected, so the caller passes
 * the selection.
 *  axis  FEATFIX_MASK_NONE: whole-block forwarding (Eq. 5, the default).
 *        FEATFIX_MASK_TOKENS: mask[n], n = 0 .. txt_tokens + image tokens - 1
 *        in a sample's sequence order (text first), the same for every
 *        sample of the model batch.
 *        FEATFIX_MASK_CHANNELS: mask[c], c = 0 .. hidden - 1.
 *  mask  host bytes, nonzero = forward h^f; copied (the call synchronises
 *        the context stream and drops a captured trajectory graph).
 * Only the FeatFix arm uses the mask.  Errors: INVALID_ARG for an unknown
 * axis, a null mask or a length other than the axis' size.                  */
enum { FEATFIX_MASK_NONE = 0, FEATFIX_MASK_TOKENS = 1, FEATFIX_MASK_CHANNELS = 2 };
FEATFIX_API featfix_status featfix_set_forward_mask(featfix_ctx* ctx, int axis, const unsigned char* mask, int n);

/* Host-only: per (step, block) draft order k_eff [steps*n_layers] (-1
 * where the block is exact) and weights [steps*n_layers*4] of the history
 * that block's draft reads.  Equal to featfix_plan_build's per-step values
 * for every block unless flags has FEATFIX_FLAG_SITE_UPDATES_HISTORY.        */
FEATFIX_API featfix_status featfix_plan_build_blocks(int steps, int n_layers, const int* refresh, int n_refresh,
                                         int draft_order, const featfix_site* sites, int n_sites, int mode,
                                         unsigned flags, int* k_eff, double* weights);

/* Debug capture: during later trajectories, copy block `layer`'s incoming
 * state u and its forwarded output at step `step` into dev_in / dev_out
 * (device, B_model*N_tot*C elements of the model dtype, row layout of
 * featfix_token_row).  Up to 64 captures (of either kind below); step < 0
 * clears them all.                                                           */
FEATFIX_API featfix_status featfix_debug_capture(featfix_ctx* ctx, int step, int layer, void* dev_in, void* dev_out);

/* Debug capture of the refresh history a draft reads (Eq. 2's finite
 * differences are formed from these increments): during later trajectories,
 * when block `layer` is drafted or paid-checked at step `step`, copy the
 * first min(n, K_eff + 1) increments h^f - u of its history, newest first,
 * as the block's draft reads them, into dev_slots[0..n-1] (device, each
 * B_model*N_tot*C elements of the model dtype, row layout of
 * featfix_token_row).  Nothing is copied when the block is exact at that
 * step.  1 <= n <= 4.  Errors: INVALID_ARG for a bad layer, n or pointer.    */
FEATFIX_API featfix_status featfix_debug_capture_history(featfix_ctx* ctx, int step, int layer,
                                                         void* const* dev_slots, int n);

/* Failure-detection test hook (the paper has no counterpart).  Launches, on
 * the context stream, one CTA that takes tensor memory as the tensor-core
 * GEMM does and then waits, with the GEMM's bounded wait, on an mbarrier
 * that nothing arrives on.  After limit_ns (1 us .. 1 s) the wait gives up,
 * raises the watchdog flag a stuck GEMM or attention kernel raises, and the
 * CTA frees its tensor memory and returns: nothing traps and the context
 * stays usable.  The next featfix_get_log then reports FEATFIX_ERR_CUDA
 * (and clears the flag).  Errors: INVALID_ARG for a limit out of range.     */
FEATFIX_API featfix_status featfix_debug_watchdog_probe(featfix_ctx* ctx, unsigned long long limit_ns);

/* Run the exact block B_l(u; t_step, c) (Eq. 1) on a caller state: dev_in,
 * dev_out as for featfix_debug_capture, dev_cond as for featfix_step.
 * Requires a schedule (for t_step).  Ordered on the context stream.         */
FEATFIX_API featfix_status featfix_debug_block(featfix_ctx* ctx, int step, int layer, const void* dev_in,
                                   void* dev_out, const void* dev_cond);

/* Row of token n (0 <= n < N_txt + N_img, text first) of model-batch sample
 * b in the library's token layout.  Text rows of all samples come first
 * (b*N_txt + n), then image rows (B_model*N_txt + b*N_img + n - N_txt).   */
FEATFIX_API long long featfix_token_row(const featfix_model_desc* desc, int b, int n);

/* Kernel timing: when on, launches of the kernel class `kclass`
 * (FEATFIX_KCLASS_*) are bracketed by CUDA events on the context stream;
 * featfix_kernel_time returns the summed duration (ms) and launch count
 * since it was switched on (synchronises the stream).                      */
enum { FEATFIX_KCLASS_GEMM = 0, FEATFIX_KCLASS_ATTENTION = 1, FEATFIX_KCLASS_DRAFT = 2,
       FEATFIX_KCLASS_VERIFY = 3, FEATFIX_KCLASS_OTHER = 4 };
FEATFIX_API featfix_status featfix_kernel_timing(featfix_ctx* ctx, int kclass, int on);
FEATFIX_API featfix_status featfix_kernel_time(featfix_ctx* ctx, int kclass, double* ms, long long* launches,
                                   double* work);

/* Number of kernels this library has launched in the calling process so far
 * (all contexts and op calls); a diagnostic for launch accounting.         */
FEATFIX_API long long featfix_launch_count(void);

FEATFIX_API const char* featfix_last_error(const featfix_ctx* ctx);
FEATFIX_API const char* featfix_status_string(featfix_status s);
FEATFIX_API void featfix_destroy(featfix_ctx* ctx);

#ifdef __cplusplus
}
#endif
#endif /* FEATFIX_H */
