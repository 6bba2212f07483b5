// internal.h -- host-side launch interfaces shared by the library's .cu files.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "../../include/ff.h"

namespace ff {

// ---- error reporting (thread-local message behind ff_last_error) --------
int set_error(int code, const char* fmt, ...);
int check_launch(const char* what);       // FF_ERR_CUDA if the last launch failed
int* device_status_ptr();                  // address of the current device's status word
int num_sms();                             // SM count of the current device

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Return the status of a library call from the enclosing function if it failed.
#define FF_TRY(expr)                \
    do {                            \
        const int rc_ = (expr);     \
        if (rc_ != FF_OK) return rc_; \
    } while (0)

// Configuration of a DiT handle (its struct is private to dit.cu).
const ff_dit_config& model_config(const ff_dit* m);

// ---- optional launch timing (ff_prof_*): RAII scope around one launch ----
struct ProfScope {
    ProfScope(cudaStream_t s, const char* name, double flops, double bytes);
    ~ProfScope();
    int slot;
    cudaStream_t stream;
};

// ---- tensor maps ---------------------------------------------------------
// 2-D bf16 row-major matrix [rows, cols] with leading dimension ld
// (elements), box = box_rows x 64 columns, 128-byte swizzle, zero fill.
int make_tmap_bf16(CUtensorMap* tm, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_rows);
// 2-D fp32 matrix, box = box_rows x 32 columns (128 bytes), 128-byte swizzle.
int make_tmap_f32_sw128(CUtensorMap* tm, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_rows);
// GEMM output tile store map: box = 32 rows x 32 columns of fp32 (128-byte
// swizzle) or bf16 (64-byte swizzle).
int make_tmap_out(CUtensorMap* tm, const void* base, int64_t rows, int64_t cols, int64_t ld, bool f32);

// ---- GEMM: D[M, N] = A[M, K] B[N, K]^T with a fused epilogue --------------
enum GemmAct { ACT_NONE = 0, ACT_GELU = 1, ACT_SILU = 2 };
enum GemmEpi { EPI_STORE = 0, EPI_GATED_RESIDUAL = 1 };

struct GemmEpilogue {
    int epi = EPI_STORE;
    int act = ACT_NONE;
    int act_from = 0;                  // activation applies to columns >= act_from
    int out_f32 = 0;                   // EPI_STORE: fp32 (1) or bf16 (0) output
    const __nv_bfloat16* bias = nullptr;  // [N] or null
    void* out0 = nullptr;              // columns [0, split_n)
    int64_t ld0 = 0;
    void* out1 = nullptr;              // columns [split_n, N) -> out1[:, n - split_n + col1]
    int64_t ld1 = 0;
    int col1 = 0;
    int split_n = 1 << 30;
    // EPI_GATED_RESIDUAL: resid[m, n] += gate[(m / rows_per_sample) * ld_gate + n] * (acc + bias);
    // gate == nullptr means a plain residual update (gate 1)
    float* resid = nullptr;
    int64_t ld_resid = 0;
    const float* gate = nullptr;
    int64_t ld_gate = 0;
    int rows_per_sample = 1;
    // Fused per-head RMSNorm (+ RoPE) of the q and k columns [0, qk_cols) of
    // a bf16 EPI_STORE output (qk_cols = 2H, head width head_dim; q scale for
    // columns < qk_cols / 2, k scale above).  Rows >= rope_row0 are latent
    // tokens (row - rope_row0) % n_img of the (grid_f, grid_h, grid_w) grid
    // and are rotated with the cos/sin table rope_cs (see rope_table); rows
    // below rope_row0 are text tokens at position 0.
    // Few-row products run on the GEMV kernel in passes of 8 rows whatever M
    // is, so each row's result does not depend on how many rows share the
    // launch (batch-invariant time embedding and modulation).
    int rows_gemv = 0;
    int qk_cols = 0;
    int head_dim = 0;
    const __nv_bfloat16* q_scale = nullptr;
    const __nv_bfloat16* k_scale = nullptr;
    const float2* rope_cs = nullptr;   // null: no rotation at all
    int rope_row0 = 0, n_img = 1, grid_f = 1, grid_h = 1, grid_w = 1;
    int axes0 = 0, axes1 = 0, axes2 = 0;
};

// cos / sin of every (axis, position, pair) rotation angle pos * theta^(-2j/a):
// table[axis0: f * a0/2 + j | axis1: F a0/2 + r * a1/2 + j | axis2: ... + c * a2/2 + j]
int rope_table_size(int grid_f, int grid_h, int grid_w, int a0, int a1, int a2);
int rope_table(float2* table, int grid_f, int grid_h, int grid_w, int a0, int a1, int a2, float theta,
               cudaStream_t stream);

int gemm_bf16(const void* A, int64_t lda, const void* B, int64_t ldb, int M, int N, int K,
              const GemmEpilogue& epi, cudaStream_t stream);

// One or two independent GEMMs in a single persistent launch (tiles of the
// first problem, then of the second).
// D[M, N] = op(A) op(B) with A stored [M, K] (a_mn = 0, K contiguous) or
// [K, M] (a_mn = 1, M contiguous), and B stored [N, K] (b_mn = 0: D = A B^T,
// the nn.Linear product) or [K, N] (b_mn = 1: D = A B).  Leading dimensions
// are those of the stored layouts.
struct GemmArgs {
    const void* A; int64_t lda;
    const void* B; int64_t ldb;
    int M, N, K;
    GemmEpilogue epi;
    int a_mn = 0, b_mn = 0;
};
int gemm_bf16_group(const GemmArgs* problems, int n, cudaStream_t stream);

// ---- elementwise / row kernels -------------------------------------------
// Row r of x (fp32 [rows, H]) belongs to segment txt if r < rows_txt, else img;
// sample b = (r - seg_start) / tokens_per_sample.  out = LN(x) (1 + scale) + shift.
struct LnModArgs {
    const float* x; int64_t ldx;
    __nv_bfloat16* out; int64_t ldo;
    int rows, H;
    int rows_txt, n_txt, n_img;        // segment split and tokens per sample
    const float* mods; int64_t ld_mods;
    int shift_txt, scale_txt, shift_img, scale_img;  // column offsets into mods
    // affine LayerNorm instead of modulation when aff_w is set: LN(x) w + b
    const __nv_bfloat16* aff_w = nullptr;
    const __nv_bfloat16* aff_b = nullptr;
};
int ln_modulate(const LnModArgs& a, cudaStream_t stream);

// In-place per-head RMSNorm plus (optionally) RoPE on up to two column
// blocks ("q" at col[0], "k" at col[1]; -1 skips a block) of a bf16 buffer
// [rows, ld].  Rows < rows_txt are text tokens (position 0: no rotation).
struct QkNormRopeArgs {
    __nv_bfloat16* qkv; int64_t ld;
    int rows, heads, head_dim;
    int rows_txt, n_img;               // rows >= rows_txt are image tokens
    int grid_f, grid_h, grid_w;
    int axes0, axes1, axes2;
    float theta;
    const __nv_bfloat16* q_scale_txt; const __nv_bfloat16* k_scale_txt;
    const __nv_bfloat16* q_scale_img; const __nv_bfloat16* k_scale_img;
    int col[2] = {0, -1};
    int rope = 1;
};
int qk_norm_rope(const QkNormRopeArgs& a, cudaStream_t stream);

// Joint attention over [text; image] token segments of each sample.
struct AttnSegment {
    const __nv_bfloat16* qkv; int64_t ld;  // q at col 0, k at col H, v at col 2H (row = token)
    __nv_bfloat16* out; int64_t ldo;       // output row = token, head h at col h*d
    int n;                                 // tokens per sample in this segment
};
int attention(const AttnSegment& s0, const AttnSegment& s1, int B, int heads, int head_dim, int H,
              cudaStream_t stream);

// General form: queries from up to two query segments, keys/values from up
// to two key/value segments (concatenated per sample), head h of q / k / v
// at columns q_col / k_col / v_col + h * d of its buffer.  Joint attention
// uses the same buffers for both; cross-attention uses image queries and
// text keys/values.
struct AttnQuerySeg { const __nv_bfloat16* buf; int64_t ld; int n; __nv_bfloat16* out; int64_t ldo; };
struct AttnKvSeg { const __nv_bfloat16* buf; int64_t ld; int n; };
struct AttnSpec {
    AttnQuerySeg q[2];
    AttnKvSeg kv[2];
    int q_col, k_col, v_col;
    int B, heads, head_dim;
    // optional: the per-row log-sum-exp of the scaled scores, in base 2
    // (lse2 = log2 sum_j 2^(s_j log2(e) / sqrt(d))), kept for the backward:
    // lse[(b * heads + h) * attn_lse_rows(q0, q1) + (seg ? pad128(q0) : 0) + row]
    float* lse = nullptr;
};
inline int attn_pad128(int n) { return (n + 127) / 128 * 128; }
inline int attn_lse_rows(int n0, int n1) { return attn_pad128(n0) + attn_pad128(n1); }
int attention_general(const AttnSpec& a, cudaStream_t stream);

// Backward of joint attention (d = 128): from dO (bf16, the layout of the
// forward's output) and the forward's lse, the gradients of q, k and v are
// written into dqkv buffers laid out like the qkv inputs.  ws holds
// D = rowsum(dO * O) in the lse layout (attention_backward_ws_bytes).
struct AttnBwdSeg {
    const __nv_bfloat16* qkv; int64_t ld;   // q, k, v at columns 0, H, 2H
    const __nv_bfloat16* o;                  // forward output, row pitch ldo
    const __nv_bfloat16* dout;               // its gradient, row pitch ldo
    int64_t ldo;
    __nv_bfloat16* dqkv; int64_t ldd;        // dq, dk, dv at columns 0, H, 2H
    int n;
};
size_t attention_backward_ws_bytes(int B, int heads, int n0, int n1);
int attention_backward(const AttnBwdSeg& s0, const AttnBwdSeg& s1, int B, int heads, int head_dim,
                       const float* lse, void* ws, size_t ws_bytes, cudaStream_t stream);

// mods[b, l*6H + j] = e0[b, j] + bias_l[j] (bias_l = bias0 + l*stride), and
// mods[b, L*6H + j] = e[b, j % H] + fbias[j] for j < 2H (WAN modulation).
int wan_modulation(const float* e, const float* e0, const __nv_bfloat16* bias0, int64_t stride, int L,
                   const __nv_bfloat16* fbias, int B, int H, float* mods, int64_t ld_mods, cudaStream_t stream);

int timestep_embed(const float* t, int B, int dim, __nv_bfloat16* out, cudaStream_t stream);
int f32_to_bf16(const float* in, __nv_bfloat16* out, int64_t n, cudaStream_t stream);

}  // namespace ff
