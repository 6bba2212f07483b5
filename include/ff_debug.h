/*
 * ff_debug.h -- per-kernel entry points of the velocity path, exported so the
 * parity tests can check each stage on identical inputs (the composed call is
 * ff_dit_velocity in ff.h).  Same conventions as ff.h: device pointers,
 * caller-owned memory, int status, work enqueued on `stream`.
 */
#ifndef FF_DEBUG_H
#define FF_DEBUG_H

#include "ff.h"

#ifdef __cplusplus
extern "C" {
#endif

#define FF_ACT_NONE 0
#define FF_ACT_GELU 1   /* tanh form: x/2 (1 + tanh(sqrt(2/pi)(x + 0.044715 x^3))) */
#define FF_ACT_SILU 2   /* x / (1 + exp(-x)) */

/* out[m, n] = act(sum_k A[m, k] B[n, k] + bias[n]) on the tcgen05 GEMM.
 * A: bf16 [M, lda]; B: bf16 [N, ldb] (nn.Linear weight); bias: bf16 [N] or
 * NULL; out: fp32 (out_f32 = 1) or bf16 [M, ldo].  N % 32 == 0, K % 8 == 0,
 * lda, ldb multiples of 8. */
int ff_debug_gemm(int M, int N, int K, const void* A, int64_t lda, const void* B, int64_t ldb,
                  const void* bias, int act, int out_f32, void* out, int64_t ldo, cudaStream_t stream);

/* resid[m, n] += gate[(m / rows_per_sample) * ld_gate + n] * (sum_k A[m,k] B[n,k] + bias[n])
 * (the adaLN gated residual of the projection and MLP-out GEMMs).
 * resid: fp32 [M, ld_resid]; gate: fp32. */
int ff_debug_gemm_gated(int M, int N, int K, const void* A, int64_t lda, const void* B, int64_t ldb,
                        const void* bias, float* resid, int64_t ld_resid, const float* gate, int64_t ld_gate,
                        int rows_per_sample, cudaStream_t stream);

/* Joint attention of B samples over [segment 0 (n0 tokens); segment 1 (n1
 * tokens)].  qkv_s: bf16 rows = tokens (sample-major), q at column h*d, k at
 * hidden + h*d, v at 2*hidden + h*d, row pitch ld_s; out_s: bf16 rows =
 * tokens, head h at column h*d, pitch ldo_s.  hidden = heads * head_dim. */
int ff_debug_attention(int B, int heads, int head_dim, int n0, const void* qkv0, int64_t ld0, void* out0,
                       int64_t ldo0, int n1, const void* qkv1, int64_t ld1, void* out1, int64_t ldo1,
                       cudaStream_t stream);

/* Which variant of the attention kernel every later forward launch takes,
 * process-wide (for tests): 0 the launcher's own choice by item count and
 * length, 1 the persistent one (one CTA per SM) without the split of the
 * last round's items, 2 one 256-row query block per CTA, 3 the persistent
 * one with the split wherever the launch has a scratch and its last round
 * is at most half full.  Returns the previous setting; FF_ERR_INVALID_ARG
 * (and no change) for other values.  Variants 0, 1 and 2 give bit-identical
 * output when no split is taken; a split launch agrees to fp32 rounding. */
int ff_debug_attention_launch(int mode);

/* The attention launcher's plan for `items` work items (256-row query
 * blocks) of `steps` K/V steps each on a GPU of `sms` SMs, with (have_ws !=
 * 0) or without the split scratch, under launch mode `mode` (as
 * ff_debug_attention_launch).  Host arithmetic only: nothing is launched
 * and no GPU is needed.  Writes (host pointers) *persistent (1: one CTA per
 * SM runs a strided share of the items; 0: one item per CTA), *grid (CTAs),
 * and *split_first, *split_n: items split_first .. split_first + split_n - 1
 * run as two halves of their K/V steps on CTAs 0 .. 2 split_n - 1 (split_n
 * = 0: no split).  FF_ERR_INVALID_ARG for items, sms or steps <= 0, a mode
 * outside 0-3 or a null pointer. */
int ff_debug_attention_plan(int64_t items, int sms, int steps, int have_ws, int mode, int* persistent,
                            int64_t* grid, int64_t* split_first, int64_t* split_n);

/* out[r] = LN(x[r]) * (1 + mods[b, scale_off:]) + mods[b, shift_off:] for
 * rows r of x (fp32 [rows, H]); b = r / tokens_per_sample; out bf16 [rows, H]. */
int ff_debug_ln_modulate(int rows, int H, const float* x, const float* mods, int64_t ld_mods, int shift_off,
                         int scale_off, int tokens_per_sample, void* out, cudaStream_t stream);

/* In-place RMSNorm (scales q_scale, k_scale: bf16 [head_dim]) and RoPE of the
 * q and k parts of qkv (bf16 [rows, ld], q at 0, k at heads*head_dim).  Rows
 * < rows_txt are text tokens at position 0; row r >= rows_txt is image token
 * (r - rows_txt) % (f*h*w) of the (f, h, w) grid. */
int ff_debug_qk_norm_rope(int rows, int rows_txt, int heads, int head_dim, void* qkv, int64_t ld,
                          const void* q_scale, const void* k_scale, int grid_f, int grid_h, int grid_w,
                          const int* rope_axes, float rope_theta, cudaStream_t stream);

/* Fixed-order column sums of per-chunk partials (the gradient reductions of
 * the training pass), n jobs run as launches of up to 8.  Job i sums columns
 * [0, ncols[i]) of the fp32 chunk rows at part + part_off[i] (row pitch
 * ld_part[i] floats) over one or two spans of rows: span s starts at row
 * first[2i + s] and has count[2i + s] rows (count[2i + 1] == 0: one span).
 * per_sample[i] != 0: sample b < B sums rows first + b count .. of each span
 * into out + out_off[i] + b ld_out[i]; else all count rows of each span into
 * out + out_off[i].  Each sum is taken in fp64 in a fixed order that does not
 * depend on the other jobs of the launch.  The job arrays are host memory,
 * read before the call returns; part and out are device memory. */
int ff_debug_reduce_chunks(int n, int B, const float* part, float* out, const int64_t* part_off,
                           const int64_t* ld_part, const int* ncols, const int* first, const int* count,
                           const int* per_sample, const int64_t* out_off, const int64_t* ld_out, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* FF_DEBUG_H */
