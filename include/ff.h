/*
 * ff.h -- C ABI of the GB300 (sm_103a) rollout denoising step of a
 * flow-matching DiT under Flow-GRPO-style reinforcement learning.
 *
 * The step (paper Sec. 3.1, Eq. 1 and Table 1; Sec. 2.3 "advantage
 * computation"):
 *   1. v = v_theta(x_t, t)                        ff_dit_velocity
 *   2. x_{t+dt} = Eq. 1 update, log p(x_{t+dt}|x_t) ff_sde_step_logprob
 *   3. A = group-normalised reward                 ff_group_advantage
 *   4. clipped-ratio policy loss over (b, step)    ff_grpo_loss
 * and its variants: the MixGRPO SDE window (ff_sde_schedule_window), the
 * GRPO-Guard step weights (ff_grpo_loss_weighted), multi-reward advantage
 * aggregation (ff_group_advantage_multi), and the AWM training step of
 * Sec. 3.2, Eq. 3 (ff_sample_timesteps, ff_forward_process, the velocity,
 * ff_awm_loss).
 *
 * Conventions for every entry point:
 *   - Returns an int status: FF_OK or one of the FF_ERR_* codes below.  On
 *     error nothing is launched and ff_last_error() (thread-local) says why.
 *   - Array arguments are DEVICE pointers owned by the caller, unless the
 *     comment says "host".  They must be 16-byte aligned (128-bit vector
 *     access) and must not alias unless stated.
 *   - Work is enqueued on the caller's stream; results are valid once that
 *     stream has been synchronised.  No entry point synchronises the device,
 *     and none allocates device memory: scratch space is a caller-owned
 *     workspace whose size comes from the matching *_workspace_size query.
 *   - Errors found inside a kernel (a bounded wait that ran out) set a device
 *     status word; ff_check_device_status() reads and clears it.
 */
#ifndef FF_H
#define FF_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------ */
#define FF_OK 0
#define FF_ERR_INVALID_ARG 1   /* null pointer, bad size, misalignment, bad enum */
#define FF_ERR_UNSUPPORTED 2   /* shape outside what the kernels handle        */
#define FF_ERR_WORKSPACE 3     /* workspace missing or too small               */
#define FF_ERR_CUDA 4          /* a CUDA runtime/driver call or launch failed  */
#define FF_ERR_DEVICE_CHECK 5  /* a kernel reported an error via status word   */

/* ---- enums ------------------------------------------------------------- */
#define FF_SDE_SAMPLE 0   /* draw x_next = mean + std * eps and write it     */
#define FF_SDE_EVAL 1     /* read the given x_next and only score it        */
#define FF_LP_SUM 0       /* log-prob summed over the D elements of a sample */
#define FF_LP_MEAN 1      /* ... divided by D                                */

#define FF_SCHED_FLOW_SDE 0   /* Table 1: sigma_t = eta sqrt(t/(1-t))       */
#define FF_SCHED_DANCE_SDE 1  /* Table 1: sigma_t = eta                     */
#define FF_SCHED_ODE 2        /* Table 1: sigma_t = 0                       */

#define FF_TSAMPLE_UNIFORM 0       /* Sec. 3.2 training times: t = p0 + (p1 - p0) u          */
#define FF_TSAMPLE_LOGIT_NORMAL 1  /* t = 1 / (1 + exp(-(p0 + p1 z)))                       */
#define FF_TSAMPLE_DISCRETE 2      /* t = grid[min(floor(u n), n - 1)]                      */

#define FF_AWM_SUM 0    /* Eq. 3 squared norm: sum over the D elements of a sample */
#define FF_AWM_MEAN 1   /* ... divided by D (per-element MSE)                     */

#define FF_AGG_WEIGHTED_SUM 0  /* r = sum_k w_k R_k, then group-normalise r          */
#define FF_AGG_PER_REWARD 1    /* group-normalise each R_k, then sum_k w_k A_k (GDPO) */

#define FF_A_MK 0   /* ff_gemm: A stored [M, K] */
#define FF_A_KM 1   /* ff_gemm: A stored [K, M] */
#define FF_B_NK 0   /* ff_gemm: B stored [N, K] (D = A B^T, the nn.Linear product) */
#define FF_B_KN 1   /* ff_gemm: B stored [K, N] (D = A B) */

#define FF_ARCH_MMDIT 0   /* Flux / Qwen-Image style double + single stream */
#define FF_ARCH_WAN 1     /* WAN-style video DiT: self-attn + text cross-attn + FFN */

/* Last error message of the calling thread ("" if none). */
const char* ff_last_error(void);

/* Library version, major*10000 + minor*100 + patch. */
int ff_version(void);

/* Reads and clears the device status word of the current device (0 = no
 * kernel-reported error).  Synchronises the given stream first. */
int ff_check_device_status(cudaStream_t stream, int* status_out);

/* ------------------------------------------------------------------------
 * Optional launch timing (off by default).  While enabled, every kernel the
 * library launches is bracketed by two CUDA events recorded on its stream,
 * and the record keeps the kernel's name and its algorithmic work (flops and
 * bytes that the operation must do, not what the kernel happens to move).
 * ff_prof_enable creates the events up front (host-side; no device memory);
 * launches beyond max_records are not timed.  ff_prof_read synchronises on
 * record i's end event.  Not for use under stream capture.
 * ------------------------------------------------------------------------ */
int ff_prof_enable(int max_records);
int ff_prof_disable(void);
int ff_prof_reset(void);
int ff_prof_count(int* n);
int ff_prof_read(int i, char* name, int name_cap, float* ms, double* flops, double* bytes);

/* ------------------------------------------------------------------------
 * Sampler schedule (host only).  Paper Table 1 and Eq. 1.
 *   t_out[0..n_steps]: t_k = 1 - k/n_steps, mapped by the time shift
 *     t' = shift t / (1 + (shift - 1) t) when shift != 1  (host array).
 *   sigma_out[0..n_steps-1]: sigma at each step's start time t_k; for
 *     FF_SCHED_FLOW_SDE t is clamped to t_clamp inside the square root
 *     (the formula is singular at t = 1).  Host array.
 * ------------------------------------------------------------------------ */
int ff_sde_schedule(int kind, int n_steps, double shift, double eta, double t_clamp,
                    double* t_out, double* sigma_out);

/* ------------------------------------------------------------------------
 * MixGRPO / Flow-GRPO-Fast (paper Sec. 3.1): SDE noise on the steps
 * window_start .. window_start + window_len - 1 only and the deterministic
 * ODE update elsewhere.  Same as ff_sde_schedule, with sigma_out[k] = 0
 * outside the window (an ODE step's log-prob is 0, see below).  Requires
 * 0 <= window_start and window_start + window_len <= n_steps.  Host only.
 * ------------------------------------------------------------------------ */
int ff_sde_schedule_window(int kind, int n_steps, double shift, double eta, double t_clamp,
                           int window_start, int window_len, double* t_out, double* sigma_out);

/* ------------------------------------------------------------------------
 * SDE step + Gaussian transition log-probability.  Paper Eq. 1, Table 1.
 * Time runs from 1 (noise) to 0 (data); with Delta = t - t_next > 0,
 *   mean = x - [v + sigma^2/(2t) (x + (1-t) v)] Delta,   std = sigma sqrt(Delta)
 *   SAMPLE: x_next = mean + std * eps (written);  EVAL: x_next is read.
 *   logp[b * ld] = sum_j -(x_next_j - mean_j)^2/(2 std^2) - D ln std - D/2 ln 2pi
 *   (divided by D for FF_LP_MEAN).  A sample with std == 0 (ODE step) gets
 *   x_next = mean and logp = 0.
 *
 * B samples of D fp32 elements each, row-major [B, D]; D % 4 == 0.
 *   x_t, v:      [B, D] fp32, read.
 *   eps:         [B, D] fp32, read in SAMPLE mode; may be NULL in EVAL mode.
 *   x_next:      [B, D] fp32, written (SAMPLE) or read (EVAL).  May alias x_t
 *                in SAMPLE mode (in-place update).
 *   t, t_next, sigma: [B] fp32 each (device), per-sample times and sigma;
 *                require 0 < t, t_next < t, sigma >= 0 (not checked on the
 *                host: device values).
 *   logp:        fp32, logp[b * ld] written for b < B; ld >= 1.
 *   ws:          workspace of at least ff_sde_workspace_size(B, D) bytes,
 *                16-byte aligned.  Its first 256 KiB hold ticket counters
 *                that must be ZERO before the first call that uses the
 *                workspace (cudaMemsetAsync it once after allocating); every
 *                call leaves them zero again, so a workspace zeroed once
 *                serves any number of calls of any B and D in stream order.
 *                Calls that share a workspace must not overlap on the GPU.
 * B <= 65535.  One kernel launch: every block stores a partial sum of its
 * squared residuals and the last block of each sample adds that sample's
 * partials in a fixed order, so logp is deterministic.
 * ------------------------------------------------------------------------ */
int ff_sde_workspace_size(int B, int64_t D, size_t* bytes);
int ff_sde_step_logprob(int B, int64_t D, const float* x_t, const float* v,
                        const float* eps, float* x_next, const float* t,
                        const float* t_next, const float* sigma, int mode, int reduce,
                        float* logp, int ld, void* ws, size_t ws_bytes,
                        cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Counter-based noise for SAMPLE steps (the eps of Eq. 1 drawn on the device;
 * the paper does not say where the noise comes from).  Philox4x32 with 10
 * rounds (Salmon, Moraes, Dror, Shaw, SC 2011) and the Box-Muller transform:
 * elements 4g .. 4g + 3 of sample b in stream `rng_stream` (the step index)
 * come from one call with counter (g, b, rng_stream, 0) and key (seed mod
 * 2^32, seed div 2^32).  Each output word w gives u = (floor(w / 512) + 1/2)
 * 2^-23, and the pairs (u0, u1), (u2, u3) give sqrt(-2 ln u0) (cos 2 pi u1,
 * sin 2 pi u1), sqrt(-2 ln u2) (cos 2 pi u3, sin 2 pi u3).  Any element of
 * any step is reproducible from (seed, rng_stream, b, index) alone.
 *
 * ff_philox_normal: out [B, D] fp32 (device, 16-byte aligned) = those noises.
 * ff_sde_step_logprob_philox: ff_sde_step_logprob in FF_SDE_SAMPLE mode with
 *   eps drawn inside the kernel instead of read (12 bytes per element of
 *   HBM traffic instead of 16); x_next and logp equal those of
 *   ff_sde_step_logprob given eps = ff_philox_normal(B, D, seed, rng_stream)
 *   up to the order of floating-point operations.
 * D a multiple of 4 and D / 4 < 2^32; other arguments and errors as
 * ff_sde_step_logprob.
 * ------------------------------------------------------------------------ */
int ff_philox_normal(int B, int64_t D, uint64_t seed, uint32_t rng_stream, float* out,
                     cudaStream_t stream);
int ff_sde_step_logprob_philox(int B, int64_t D, const float* x_t, const float* v,
                               float* x_next, const float* t, const float* t_next,
                               const float* sigma, uint64_t seed, uint32_t rng_stream,
                               int reduce, float* logp, int ld, void* ws, size_t ws_bytes,
                               cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Gradient of the transition log-probability in v, with x_next held fixed
 * (the training pass of Flow-GRPO, Sec. 3.1, re-scores the rollout's x_next
 * under the current velocity).  From Eq. 1, mean depends on v as
 * d mean_j / d v_j = -Delta (1 + sigma^2 (1 - t) / (2 t)), so
 *   grad_v[b, j] = grad_logp[b * ld] * (x_next_j - mean_j) / std^2
 *                  * d mean_j / d v_j   (divided by D for FF_LP_MEAN),
 * and 0 where std == 0 (no density).  Arrays as ff_sde_step_logprob (EVAL);
 * grad_logp: fp32 device, read at b * ld (e.g. a column of the
 * grad_lp_new output of ff_grpo_loss, ld = T); grad_v: [B, D] fp32,
 * written (may not alias the inputs).  No workspace.
 * ------------------------------------------------------------------------ */
int ff_sde_logprob_backward(int B, int64_t D, const float* x_t, const float* v,
                            const float* x_next, const float* t, const float* t_next,
                            const float* sigma, int reduce, const float* grad_logp, int ld,
                            float* grad_v, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * ff_sde_step_logprob_noalloc -- the SDE step + log-prob above, for callers
 * that cannot allocate device memory: for example a plug-in running inside a
 * host application that owns every device allocation itself (its own pool,
 * its own accounting), where an extra cudaMalloc would fragment that pool,
 * bypass its limits, or stall the device at a moment the host does not
 * control.  The paper has no counterpart; this is a deployment convenience.
 *
 * Same arguments and results as ff_sde_step_logprob, minus the workspace.
 * The caller still passes every input and output.  The scratch is a fixed
 * 272 KiB array built into the library (4096 ticket counters, then 65536
 * fp32 partial sums), held on every GPU that loads the library until the
 * process exits.  Limits: B <= 4096 and B * min(ceil(D / 4096), 1024) <=
 * 65536 partial sums, which holds for any D when B <= 64; larger calls are
 * rejected with FF_ERR_UNSUPPORTED and a message naming the limit, before any
 * pointer is looked at.  Nothing here calls cudaMalloc, cudaFree or any
 * other allocating routine.
 *
 * The first call on each device looks up the array's device address
 * (cudaGetSymbolAddress, with that device current) and caches it per device
 * ordinal; make that first call before any stream capture begins.  The
 * cached address belongs to the device's primary context: it is not valid
 * for a caller that drives the device through another context, and it goes
 * stale after cudaDeviceReset.  Every call on a device uses the same array.
 * The ticket counters start at zero when the library loads and every call
 * leaves them zero; the partial slots are rewritten before they are read.
 * Calls whose kernels overlap on the GPU (different streams, no ordering
 * between them) race on the array and must not be issued.
 * ------------------------------------------------------------------------ */
int ff_sde_step_logprob_noalloc(int B, int64_t D, const float* x_t, const float* v,
                                const float* eps, float* x_next, const float* t,
                                const float* t_next, const float* sigma, int mode, int reduce,
                                float* logp, int ld, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Group-relative advantage (paper Sec. 2.3, advantage computation of the
 * GRPO trainer).  Samples form contiguous groups of G (one prompt each):
 *   A[g*G + i] = (r[g*G + i] - mean_g) / (std_g + eps_A),  std_g population.
 * rewards, adv: [n_groups * G] fp32.  G in [1, 4096].  adv may alias rewards.
 * ------------------------------------------------------------------------ */
int ff_group_advantage(int n_groups, int G, const float* rewards, float eps_A,
                       float* adv, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Clipped-ratio policy loss of Flow-GRPO (paper Sec. 3.1; PPO-style clip):
 *   rho = exp(lp_new - lp_old),
 *   loss = -1/(B T) sum_{b,k} min(rho A_b, clip(rho, 1 - clip_lo, 1 + clip_hi) A_b)
 *   grad_lp_new[b,k] = -A_b rho / (B T) where the unclipped term is the
 *   minimum (ties: unclipped), else 0.
 * lp_new, lp_old: [B, T] fp32 row-major; adv: [B] fp32; loss: [1] fp32
 * (written); grad_lp_new: [B, T] fp32 or NULL.
 * ws: workspace of at least ff_grpo_loss_workspace_size(B, T) bytes,
 *   16-byte aligned.  Its first 16 bytes hold a ticket counter that must be
 *   ZERO before the first call that uses the workspace (clear it once after
 *   allocating); every call leaves it zero.  Calls sharing a workspace must
 *   not overlap on the GPU.  One kernel launch; the last block to finish
 *   adds the per-block partial sums in a fixed order (deterministic loss).
 * ------------------------------------------------------------------------ */
int ff_grpo_loss_workspace_size(int B, int T, size_t* bytes);
int ff_grpo_loss(int B, int T, const float* lp_new, const float* lp_old,
                 const float* adv, float clip_lo, float clip_hi, float* loss,
                 float* grad_lp_new, void* ws, size_t ws_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * GRPO-Guard (paper Sec. 3.1): the loss above with timestep-dependent
 * weights.  The term of step k (objective and gradient) is multiplied by
 * step_w[k]; the paper does not print the weights, so they are an input.
 *   loss = -1/(B T) sum_{b,k} step_w[k] min(rho A_b, clip(rho) A_b)
 * step_w: [T] fp32 device, not NULL (all ones gives ff_grpo_loss).  Same
 * workspace as ff_grpo_loss.
 * ------------------------------------------------------------------------ */
int ff_grpo_loss_weighted(int B, int T, const float* lp_new, const float* lp_old,
                          const float* adv, const float* step_w, float clip_lo, float clip_hi,
                          float* loss, float* grad_lp_new, void* ws, size_t ws_bytes,
                          cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Multi-reward advantage (paper Sec. 2.3, configurable advantage
 * aggregation, "weighted-sum and GDPO-style per-reward normalization").
 * K rewards per sample, R: [n_groups * G, K] fp32 row-major; w: [K] fp32
 * device; contiguous groups of G as in ff_group_advantage.
 *   FF_AGG_WEIGHTED_SUM: r_i = sum_k w_k R[i, k]; A_i = (r_i - mean_g) / (std_g + eps_A)
 *   FF_AGG_PER_REWARD:   A_i = sum_k w_k (R[i, k] - mean_g,k) / (std_g,k + eps_A)
 * (population std).  G in [1, 4096], K in [1, 64].  adv: [n_groups * G]
 * fp32, must not alias rewards.
 * ------------------------------------------------------------------------ */
int ff_group_advantage_multi(int n_groups, int G, int K, const float* rewards, const float* w,
                             int mode, float eps_A, float* adv, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Advantage Weighted Matching (paper Sec. 3.2, Eq. 3).  Time runs from 1
 * (noise) to 0 (data), as in the sampler above.
 *
 * ff_sample_timesteps -- training times t[b] from the caller's random draws
 * (Sec. 3.2: uniform, logit-normal or discrete timestep sampling):
 *   FF_TSAMPLE_UNIFORM:      t = p0 + (p1 - p0) draw,   draw = u in [0, 1)
 *   FF_TSAMPLE_LOGIT_NORMAL: t = 1 / (1 + exp(-(p0 + p1 draw))), draw = z ~ N(0, 1), p1 >= 0
 *   FF_TSAMPLE_DISCRETE:     t = grid[min(floor(draw n_grid), n_grid - 1)], draw = u
 *                            (the index is taken in fp32)
 * draw, t_out: [B] fp32 device; grid: [n_grid] fp32 device (DISCRETE only).
 *
 * ff_forward_process -- the noised input of Eq. 3:
 *   x_t[b, j] = (1 - t[b]) x0[b, j] + t[b] eps[b, j]
 * x0, eps, x_t: [B, D] fp32 row-major, 16-byte aligned, D % 4 == 0; t: [B]
 * fp32 device.  x_t may alias x0 or eps.
 *
 * ff_awm_loss -- Eq. 3 over a batch (the expectation over t and eps is the
 * batch mean):
 *   e_b = sum_j (v[b, j] - (eps[b, j] - x0[b, j]))^2  (/ D for FF_AWM_MEAN)
 *   loss = (1/B) sum_b A[b] e_b
 *   grad_v[b, j] = (2/B) A[b] (v[b, j] - (eps[b, j] - x0[b, j]))  (/ D for MEAN)
 * v, eps, x0: [B, D] fp32 (v = ff_dit_velocity(x_t, t)); adv: [B] fp32;
 * loss: [1] fp32 written; grad_v: [B, D] fp32 or NULL; err_out: [B] fp32
 * (e_b) or NULL.  ws: at least ff_awm_loss_workspace_size(B, D) bytes; the
 * two-pass reduction is deterministic.
 * ------------------------------------------------------------------------ */
int ff_sample_timesteps(int mode, int B, const float* draw, float p0, float p1,
                        const float* grid, int n_grid, float* t_out, cudaStream_t stream);
int ff_forward_process(int B, int64_t D, const float* x0, const float* eps, const float* t,
                       float* x_t, cudaStream_t stream);
int ff_awm_loss_workspace_size(int B, int64_t D, size_t* bytes);
int ff_awm_loss(int B, int64_t D, const float* v, const float* eps, const float* x0,
                const float* adv, int reduce, float* loss, float* grad_v, float* err_out,
                void* ws, size_t ws_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * DiffusionNFT loss (paper Sec. 3.2, Eq. 2):
 *   loss = (1/B) sum_b [ r_b e+_b + (1 - r_b) e-_b ],
 *   e+-_b = ||v+-_b - (eps_b - x0_b)||^2  (divided by D for FF_AWM_MEAN),
 * with the implicit positive / negative policies of the cited DiffusionNFT
 * method (the paper names them without defining them):
 *   v+ = (1 - beta) v_old + beta v,   v- = (1 + beta) v_old - beta v,
 * v the trained velocity and v_old the frozen velocity of the sampling
 * policy at the same (x_t, t).  The target eps - x0 is that of Eq. 3.
 *   v, v_old, eps, x0: [B, D] fp32 (D % 4 == 0); r: [B] fp32 reward weights
 *   in [0, 1] (device; not checked); beta > 0.
 *   loss: [1] fp32; grad_v: [B, D] fp32 dL/dv or NULL; err: [B, 2] fp32
 *   (e+_b, e-_b) or NULL.  ws: ff_nft_loss_workspace_size bytes, 8-byte
 *   aligned.  Deterministic (fixed-order fp64 sums).
 * ------------------------------------------------------------------------ */
int ff_nft_loss_workspace_size(int B, int64_t D, size_t* bytes);
int ff_nft_loss(int B, int64_t D, const float* v, const float* v_old, const float* eps,
                const float* x0, const float* r, float beta, int reduce, float* loss,
                float* grad_v, float* err, void* ws, size_t ws_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * DiT velocity v_theta(x_t, t) (the network of Eq. 1 and Eq. 3).
 *
 * Architecture (MMDiT, Flux / Qwen-Image style): timestep embedding MLP and
 * all adaLN modulations from one GEMM; patch and text embeddings; n_double
 * double-stream blocks (per-stream weights, joint attention over
 * [text; image]); n_single single-stream blocks; final LN-modulate + linear.
 * LayerNorm has no affine and eps 1e-6; q and k get a per-head RMSNorm with a
 * learned scale (eps 1e-6) and RoPE over (frame, row, col) slices of the head
 * dim (rope_axes, sum = head_dim; pair (2j, 2j+1) of a slice of width a turns
 * by pos * theta^(-2j/a)); text tokens sit at position (0, 0, 0); GELU is the
 * tanh form; attention scale is 1/sqrt(d).
 *
 * WAN-style DiT (arch FF_ARCH_WAN; n_double = number of blocks, n_single =
 * 0): text embedded by Linear-GELU-Linear; one shared projection of the
 * timestep embedding e to six H-wide vectors plus a learned per-block bias
 * gives each block's (shift, scale, gate) x 2; a block is LN-modulate ->
 * QKV -> per-head RMSNorm + 3-axis RoPE -> self-attention over the latent
 * tokens -> gated projection; affine LN -> cross-attention (RMSNorm'd q from
 * the latent tokens, RMSNorm'd k and v from the text, no RoPE) -> projection
 * added ungated; LN-modulate -> GELU MLP -> gated residual.  The final layer
 * uses shift / scale = e + a learned bias.
 *
 * Weights live in ONE caller-owned bf16 device blob; ff_dit_weight_layout
 * gives every tensor's name, element offset and shape (nn.Linear [out, in]).
 * ------------------------------------------------------------------------ */
typedef struct ff_dit_config {
    int arch;          /* FF_ARCH_MMDIT or FF_ARCH_WAN */
    int hidden;        /* H, multiple of 64 */
    int heads;         /* h */
    int head_dim;      /* d: 64 or 128; h * d == H */
    int mlp;           /* F, multiple of 64 */
    int n_double;      /* double-stream blocks (WAN: the number of blocks) */
    int n_single;      /* single-stream blocks (WAN: 0) */
    int patch_dim;     /* P, latent token width (64), multiple of 16 */
    int txt_dim;       /* D_txt, multiple of 64 */
    int n_txt;         /* N_t text tokens per sample */
    int grid_f, grid_h, grid_w;  /* latent token grid; N_i = f*h*w */
    int rope_axes[3];  /* head-dim slice per (frame, row, col); even; sum = d */
    float rope_theta;  /* 10000 */
    int time_freq_dim; /* sinusoid features of 1000 t (256), multiple of 64 */
} ff_dit_config;

typedef struct ff_tensor_desc {
    char name[64];     /* e.g. "double.0.img.qkv.w" */
    int64_t offset;    /* in bf16 elements from the blob start (multiple of 64) */
    int ndim;          /* 1 or 2 */
    int64_t shape[2];  /* [out, in] for matrices, [n] for vectors */
} ff_tensor_desc;

typedef struct ff_dit ff_dit;

/* Fills out[0..min(capacity, count)-1] (out may be NULL to query), sets
 * *count and *total_elems (blob size in bf16 elements). */
int ff_dit_weight_layout(const ff_dit_config* cfg, ff_tensor_desc* out, int capacity,
                         int* count, int64_t* total_elems);

/* Validates cfg and records the blob pointer (no copy, no device
 * allocation).  The blob must stay alive and unchanged until destroy. */
int ff_dit_create(const ff_dit_config* cfg, const void* weights_dev, ff_dit** out);
int ff_dit_destroy(ff_dit* model);

/* Whether the model's attention launches may split the query blocks of
 * their last, at most half-full round over the SMs into two halves of the
 * keys (see ff_attention_forward's ws): on = 1 (the default) or 0.  A split
 * block's output agrees with the unsplit one to fp32 rounding, and which
 * blocks split depends on the batch size, so with on = 1 a sample's
 * velocity can differ in its last bits between calls on different batches.
 * With on = 0 a sample's velocity (and every training-pass result) is bit
 * for bit independent of the other samples in the batch.  Applies to the
 * velocity, rollout and training entries; set it before a training
 * pass's forward and keep it until its backward.  The workspace sizes do
 * not depend on it.  Other values of on: FF_ERR_INVALID_ARG. */
int ff_dit_set_attention_split(ff_dit* model, int on);

/* Workspace bytes for a velocity call on a batch of B samples. */
int ff_dit_workspace_size(const ff_dit* model, int B, size_t* bytes);

/* v_out[b, n, :] = v_theta(x_t[b], t[b], txt[b]).
 *   x_t:   [B, N_i, P] fp32 latent tokens (row-major grid order)
 *   txt:   [B, N_t, D_txt] bf16 cached text embeddings
 *   t:     [B] fp32 times in (0, 1]
 *   v_out: [B, N_i, P] fp32 (must not alias x_t)
 *   ws:    at least ff_dit_workspace_size(model, B) bytes, 256-byte aligned */
int ff_dit_velocity(const ff_dit* model, int B, const float* x_t, const void* txt,
                    const float* t, float* v_out, void* ws, size_t ws_bytes,
                    cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Training pass of the velocity network (MMDiT and WAN-style models): the
 * forward every GRPO-style trainer runs "again for training" (Sec. 1) and
 * its gradient, for the policy losses of Sec. 3 (the Flow-GRPO loss through
 * ff_sde_logprob_backward, AWM's Eq. 3 through ff_awm_loss's dL/dv).
 *
 * ff_dit_forward_train: the same computation as ff_dit_velocity (same
 *   arguments, bit-identical v_out) that also keeps, in ws, every activation
 *   the backward reads.  ws: ff_dit_train_workspace_size bytes, 256-byte
 *   aligned; it must stay untouched until the matching ff_dit_backward.
 * ff_dit_backward: from dv = dL/dv ([B, N_i, P] fp32, device) to
 *   grad: fp32 device blob of ff_dit_weight_layout's total_elems elements,
 *     element offsets as in the weight blob; every element of every tensor
 *     is overwritten with dL/dtheta (the padding between tensors is not
 *     touched);
 *   dx_t: [B, N_i, P] fp32 dL/dx_t, or NULL.
 *   txt must hold the same text embeddings as in the forward.  Every sum
 *   over tokens runs in a fixed order: the result is deterministic.
 * Requires B N_t and B N_i multiples of 8.  The workspace holds about
 * R (30 H + 4 F) bytes per double-stream block and R (22 H + 4 F) per
 * single-stream block, R = B (N_t + N_i), plus scratch; per WAN block
 * R_i (42 H + 4 F) + 8 R_t H bytes (R_i = B N_i, R_t = B N_t).
 * ------------------------------------------------------------------------ */
/* Recompute mode of the training pass (on = 1 or 2; 0 stores every
 * activation): ff_dit_forward_train keeps every block's input residual (fp32,
 * 4 H bytes per residual row) and the backward re-runs block l's forward into
 * one shared activation set (one per block kind) just before that block's
 * backward.  on = 1 also keeps the self-attention output of every WAN block
 * and the joint-attention output of every double-stream MMDiT block (O and
 * its low part in bf16 and lse: 4 H + 4 heads bytes per query row), and the
 * re-run skips that attention, the most expensive kernel of a block; on = 2
 * keeps the block inputs only and re-runs everything.  The gradient is
 * bit-identical to the stored-activation pass in both modes (every kernel is
 * deterministic).  Other values of on: FF_ERR_INVALID_ARG.  Set it before ff_dit_train_workspace_size and keep it
 * unchanged until the matching ff_dit_backward: ff_dit_backward returns
 * FF_ERR_INVALID_ARG when the mode differs from that of the model's latest
 * ff_dit_forward_train (or when there was none). */
int ff_dit_set_train_recompute(ff_dit* model, int on);
int ff_dit_train_workspace_size(const ff_dit* model, int B, size_t* bytes);
int ff_dit_forward_train(const ff_dit* model, int B, const float* x_t, const void* txt,
                         const float* t, float* v_out, void* ws, size_t ws_bytes,
                         cudaStream_t stream);
int ff_dit_backward(const ff_dit* model, int B, const void* txt, const float* dv, float* grad,
                    float* dx_t, void* ws, size_t ws_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * bf16 GEMM with fp32 accumulation on the tcgen05 kernels of the velocity:
 *   out[M, N] = act(op(A) op(B) + bias),  op(A) [M, K], op(B) [K, N]
 * a_layout FF_A_MK: A stored [M, K] (lda >= K); FF_A_KM: A stored [K, M]
 * (lda >= M).  b_layout FF_B_NK: B stored [N, K] (ldb >= K); FF_B_KN: B
 * stored [K, N] (ldb >= N).  For a Linear y = x W^T (W [N_out, N_in]) on T
 * tokens, the training backward (the gradient pass that follows the rollout
 * in Flow-GRPO, Sec. 3.1) needs
 *   forward      y  = x W^T:   A = x  [T, N_in]  (MK), B = W [N_out, N_in] (NK)
 *   input grad   dx = dy W:    A = dy [T, N_out] (MK), B = W                (KN)
 *   weight grad  dW = dy^T x:  A = dy [T, N_out] (KM), B = x [T, N_in]      (KN)
 * bias: [N] bf16 or NULL; act: FF_ACT_NONE / GELU / SILU; out: bf16
 * (out_f32 = 0) or fp32 [M, N] with ldo.  K and every leading dimension a
 * multiple of 8, N a multiple of 32, bases 16-byte aligned.
 * ------------------------------------------------------------------------ */
int ff_gemm(int M, int N, int K, const void* A, int64_t lda, int a_layout, const void* B,
            int64_t ldb, int b_layout, const void* bias, int act, int out_f32, void* out,
            int64_t ldo, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Joint attention of the velocity network with its backward (the training
 * pass after the rollout, Sec. 3.1).  Per sample and head h, over the joint
 * token sequence [segment 0; segment 1] (text; image):
 *   O = softmax(Q K^T / sqrt(d)) V,   q, k, v of head h at columns h d,
 *   H + h d, 2H + h d of the qkv buffers (H = heads * d), O at column h d.
 * ff_attention_forward also writes lse (fp32, [B, heads, L]) with
 * L = ff_attention_lse_rows(n0, n1) = pad128(n0) + pad128(n1): the base-2
 * log-sum-exp of the scaled scores of segment-0 row r at r and of segment-1
 * row r at pad128(n0) + r (padding rows are not written).
 * ff_attention_backward (head_dim 64 or 128) takes O, its gradient dO (same
 * layout and pitch ldo) and lse, and writes dq, dk, dv into dqkv buffers laid
 * out like qkv (columns h d, H + h d, 2H + h d; pitch ldd; other columns are
 * not touched).  ws: ff_attention_backward_workspace_size bytes (holds
 * -D = -rowsum(dO * O) and a copy of -lse, each [B, heads, L]).  A segment
 * with n = 0 may pass NULL buffers.
 * ff_attention_forward's ws is optional (NULL: none): with at least
 * ff_attention_forward_workspace_size(head_dim) bytes, 16-byte aligned, a
 * launch whose work items (256 query rows of one sample and head) leave the
 * last round over the SMs at most half full runs those items as two halves
 * of their keys on two SMs each and merges the halves' partial softmaxes
 * (the online-softmax rescale, exact up to rounding).  The results agree
 * with the unsplit launch to fp32 rounding, not bit for bit.  Calls that
 * share ws must not overlap on the GPU; ws needs no initial contents.
 * ------------------------------------------------------------------------ */
int ff_attention_lse_rows(int n0, int n1);
int ff_attention_forward_workspace_size(int head_dim, size_t* bytes);
int ff_attention_forward(int B, int heads, int head_dim, int n0, const void* qkv0, int64_t ld0,
                         void* out0, int64_t ldo0, int n1, const void* qkv1, int64_t ld1,
                         void* out1, int64_t ldo1, float* lse, void* ws, size_t ws_bytes,
                         cudaStream_t stream);
int ff_attention_backward_workspace_size(int B, int heads, int n0, int n1, size_t* bytes);
int ff_attention_backward(int B, int heads, int head_dim, int n0, const void* qkv0, int64_t ld0,
                          const void* out0, const void* dout0, int64_t ldo0, void* dqkv0,
                          int64_t ldd0, int n1, const void* qkv1, int64_t ld1, const void* out1,
                          const void* dout1, int64_t ldo1, void* dqkv1, int64_t ldd1,
                          const float* lse, void* ws, size_t ws_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Cross-attention of the WAN-style block (latent queries, text keys and
 * values) with its backward.  Per sample and head h:
 *   O = softmax(Q K^T / sqrt(d)) V,  q of head h at column h d of the query
 *   rows (nq per sample, pitch ldq), k at column h d and v at H + h d of the
 *   key / value rows (nk per sample, pitch ldkv), O at column h d (pitch ldo).
 * ff_cross_attention_forward optionally writes lse (fp32, [B, heads,
 * ff_attention_lse_rows(nq, 0)], base 2, as ff_attention_forward).
 * ff_cross_attention_backward (head_dim 64 or 128) takes O, dO (pitch ldo)
 * and lse and writes dq (head h at column h d, pitch lddq) and dk | dv (head
 * h at columns h d and H + h d, pitch lddkv); ws:
 * ff_attention_backward_workspace_size(B, heads, nq, 0) bytes.  nq, nk > 0;
 * pitches multiples of 8 elements, buffers 16-byte aligned.
 * ------------------------------------------------------------------------ */
int ff_cross_attention_forward(int B, int heads, int head_dim, int nq, const void* q, int64_t ldq, int nk,
                               const void* kv, int64_t ldkv, void* out, int64_t ldo, float* lse,
                               cudaStream_t stream);
int ff_cross_attention_backward(int B, int heads, int head_dim, int nq, const void* q, int64_t ldq,
                                const void* out, const void* dout, int64_t ldo, void* dq, int64_t lddq,
                                int nk, const void* kv, int64_t ldkv, void* dkv, int64_t lddkv,
                                const float* lse, void* ws, size_t ws_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Trajectory sampling (paper Sec. 3.1: the SDE rollout that Flow-GRPO's
 * policy gradient scores, "repeated forward passes for trajectory
 * sampling").  S denoise steps; at step k = 0 .. S-1, for every sample:
 *   v = v_theta(x_k, t_k);  x_{k+1} = Eq. 1 step from t_k to t_{k+1} with
 *   sigma_k and noise eps[k] (ff_sde_step_logprob, SAMPLE mode);
 *   logp[b * S + k] = log p(x_{k+1} | x_k).
 * A step with sigma_k == 0 is an ODE step (log-prob 0), so MixGRPO windows
 * come from ff_sde_schedule_window.
 *   x:     [B, N_i, P] fp32: x_0 on entry, x_S on return (in place).
 *   txt:   [B, N_t, D_txt] bf16 text embeddings (as ff_dit_velocity).
 *   t:     [S + 1] fp32 device, the shared time grid (t_0 > ... > t_S > 0 is
 *          not checked: device values); sigma: [S] fp32 device.
 *   eps:   [S, B, N_i, P] fp32 device noise.
 *   traj:  [S + 1, B, N_i, P] fp32 device (x_0 .. x_S kept, the states the
 *          training pass re-scores) or NULL.
 *   logp:  [B, S] fp32 device, per-step log-probs of every sample.
 *   reduce: FF_LP_SUM or FF_LP_MEAN.
 *   ws:    at least ff_rollout_workspace_size(model, B, S) bytes, 256-byte
 *          aligned (holds the velocity workspace, v and the per-step times).
 * Nothing synchronises, so the call can be captured in a CUDA graph (with
 * the launch timer off).
 * ------------------------------------------------------------------------ */
int ff_rollout_workspace_size(const ff_dit* model, int B, int S, size_t* bytes);
int ff_rollout(const ff_dit* model, int B, int S, float* x, const void* txt, const float* t,
               const float* sigma, const float* eps, float* traj, float* logp, int reduce,
               void* ws, size_t ws_bytes, cudaStream_t stream);
/* ff_rollout with the noise drawn on the device: step k uses
 * ff_philox_normal's noise of (seed, rng_stream = k), inside the SDE kernel
 * (no eps buffer; the trajectory is reproducible from the seed alone).
 * Equal to ff_rollout given eps[k] = ff_philox_normal(B, D, seed, k). */
int ff_rollout_philox(const ff_dit* model, int B, int S, float* x, const void* txt, const float* t,
                      const float* sigma, uint64_t seed, float* traj, float* logp, int reduce,
                      void* ws, size_t ws_bytes, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* FF_H */
