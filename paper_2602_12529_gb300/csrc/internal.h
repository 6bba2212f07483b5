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

// Configuration, weights, parameter offsets (elements into the weight blob,
// -1 if absent) and modulation width of a DiT handle (its struct is private
// to dit.cu).
const ff_dit_config& model_config(const ff_dit* m);
const __nv_bfloat16* model_weights(const ff_dit* m);
int64_t model_offset(const ff_dit* m, const char* name);
int64_t model_mod_width(const ff_dit* m);
int model_train_recompute(const ff_dit* m);
int model_attention_split(const ff_dit* m);   // 0: the attention launches get no split scratch
// The training forward records its recompute mode on the handle; the
// backward refuses to run in another mode (the workspace layouts differ).
void model_note_forward_train(const ff_dit* m);
int model_forward_train_mode(const ff_dit* m);

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
    float* resid_out = nullptr;        // updated residual written here (same ld) instead of in place
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
    // Pre-activation copy for the training forward: when aux is set, every
    // column n of acc + bias is also stored as bf16 at aux[row * ld_aux + n]
    // before the activation, the QK norm or the gate is applied.
    __nv_bfloat16* aux = nullptr;
    int64_t ld_aux = 0;
    // Activation backward for input-gradient products: when gelu_pre is set,
    // columns n >= act_from of the product are multiplied by
    // GELU'(gelu_pre[row * ld_pre + n - act_from]), the forward's
    // pre-activation values (EPI_STORE, no activation).
    const __nv_bfloat16* gelu_pre = nullptr;
    int64_t ld_pre = 0;
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
// A weight-gradient product dW[M, N] = dy^T x over K token rows (dy [K, M],
// x [K, N], both row-major) into fp32 out (pitch N).
inline GemmArgs gemm_wgrad(const void* dy, int64_t lddy, const void* x, int64_t ldx, int M, int N, int K, float* out) {
    GemmArgs g{dy, lddy, x, ldx, M, N, K, GemmEpilogue{}};
    g.a_mn = 1;
    g.b_mn = 1;
    g.epi.out_f32 = 1;
    g.epi.out0 = out;
    g.epi.ld0 = N;
    return g;
}
// An input-gradient product dx[M, N] = dy[M, K] W[K, N] (W the forward's
// [out, in] weight read as an MN-major B operand); the caller sets the output.
inline GemmArgs gemm_dgrad(const void* dy, int64_t lddy, const void* w, int M, int N, int K) {
    GemmArgs g{dy, lddy, w, N, M, N, K, GemmEpilogue{}};
    g.b_mn = 1;
    return g;
}

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
    // optional (training): O - bf16(O) rounded to bf16, laid out like out
    // with row pitch ldo_lo; out + out_lo carries O to about 16 bits
    __nv_bfloat16* out_lo = nullptr; int64_t ldo_lo = 0;
};
int attention(const AttnSegment& s0, const AttnSegment& s1, int B, int heads, int head_dim, int H,
              cudaStream_t stream, float* lse = nullptr, void* split_ws = nullptr, size_t split_ws_bytes = 0);

// General form: queries from up to two query segments, keys/values from up
// to two key/value segments (concatenated per sample), head h of q / k / v
// at columns q_col / k_col / v_col + h * d of its buffer.  Joint attention
// uses the same buffers for both; cross-attention uses image queries and
// text keys/values.
struct AttnQuerySeg {
    const __nv_bfloat16* buf; int64_t ld; int n; __nv_bfloat16* out; int64_t ldo;
    __nv_bfloat16* out_lo = nullptr; int64_t ldo_lo = 0;   // optional low part of O (see AttnSegment)
};
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
    // optional scratch of attention_split_ws_bytes(head_dim) bytes (16-byte
    // aligned, not shared by launches that overlap on the GPU): lets a
    // persistent launch whose last round is at most half full split those
    // items' K/V steps over two CTAs each.  Without it the launch is unsplit.
    void* split_ws = nullptr;
    size_t split_ws_bytes = 0;
};
size_t attention_split_ws_bytes(int head_dim);
inline int attn_pad128(int n) { return (n + 127) / 128 * 128; }
inline int attn_lse_rows(int n0, int n1) { return attn_pad128(n0) + attn_pad128(n1); }
int attention_general(const AttnSpec& a, cudaStream_t stream);
// forward launch variant for tests: 0 automatic, 1 persistent without the
// split, 2 one item per CTA, 3 persistent with the split where it applies;
// returns the previous
int attention_launch_override(int mode);

// Backward of joint attention (d = 64 or 128): from dO (bf16, the layout of the
// forward's output) and the forward's lse, the gradients of q, k and v are
// written into dqkv buffers laid out like the qkv inputs.  ws holds
// -D = -rowsum(dO * O) and a copy of -lse, both in the lse layout
// (attention_backward_ws_bytes).
struct AttnBwdSeg {
    const __nv_bfloat16* qkv; int64_t ld;   // q, k, v at columns 0, H, 2H
    const __nv_bfloat16* o;                  // forward output, row pitch ldo
    const __nv_bfloat16* dout;               // its gradient, row pitch ldg (ldo when ldg = 0)
    int64_t ldo;
    __nv_bfloat16* dqkv; int64_t ldd;        // dq, dk, dv at columns 0, H, 2H
    int n;
    int64_t ldg = 0;
    // optional: the forward's low part of O (AttnSegment::out_lo); D then
    // comes from O to about 16 bits instead of bf16 O
    const __nv_bfloat16* o_lo = nullptr; int64_t ldo_lo = 0;
};
// The same for attention_general's form: query segments (q at column q_col
// of their rows, O, dO, and where dq goes) and key / value segments (k, v at
// columns k_col, v_col, and where dk, dv go); head h of dq / dk / dv at
// column h d of its destination.  lse: the forward's (AttnSpec layout over
// the query segments).
struct AttnBwdQuerySeg {
    const __nv_bfloat16* q; int64_t ld;
    int n;
    const __nv_bfloat16* o; int64_t ldo;
    const __nv_bfloat16* dout; int64_t ldg;
    __nv_bfloat16* dq; int64_t ldq;
    const __nv_bfloat16* o_lo = nullptr; int64_t ldo_lo = 0;   // optional low part of O
};
struct AttnBwdKvSeg {
    const __nv_bfloat16* kv; int64_t ld;
    int n;
    __nv_bfloat16 *dk, *dv; int64_t ldd;
};
struct AttnBwdSpec {
    AttnBwdQuerySeg q[2];
    AttnBwdKvSeg kv[2];
    int q_col, k_col, v_col;
    int B, heads, head_dim;
    const float* lse;
};
int attention_backward_general(const AttnBwdSpec& a, void* ws, size_t ws_bytes, cudaStream_t stream);
// D lives in the lse layout of the query segments (n0, n1 = query counts).
size_t attention_backward_ws_bytes(int B, int heads, int n0, int n1);
int attention_backward(const AttnBwdSeg& s0, const AttnBwdSeg& s1, int B, int heads, int head_dim,
                       const float* lse, void* ws, size_t ws_bytes, cudaStream_t stream);

// ---- DiT backward row / column kernels (backward.cu) ----------------------
// A segment is one stream's rows [row0, row0 + B * tokens), sample b at
// row0 + b * tokens; col_a / col_b are the mods columns of the vectors the
// kernel reads (gate_backward: gate at col_a; ln_modulate_backward: scale at
// col_b).  Kernels over segments cut each sample's rows into chunks of
// kBwdChunk rows (a chunk never straddles samples) and write one row of
// partial column sums per chunk: chunk index = first[seg] + b * chunks(seg) + k.
constexpr int kBwdChunk = 32;
__host__ __device__ inline int bwd_chunks(int tokens) { return (tokens + kBwdChunk - 1) / kBwdChunk; }
struct BwdSeg { int row0, tokens, col_a, col_b; };
struct BwdSegs {
    BwdSeg seg[2];
    int first[2];
    int n, B, chunks;
    int64_t rows;
};
BwdSegs bwd_segs(const BwdSeg* segs, int n, int B);
// Spans of chunk partials to add up: span i covers chunks [first, first + count)
// (all samples), or with a per-sample reduction sample b's chunks
// [first + b * count, first + (b + 1) * count).
struct ChunkSpans { int first[2], count[2], n; };

// Through x' = x + gate y: dy = bf16(g gate); part[c * 2H + j] = sum g y,
// part[c * 2H + H + j] = sum g gate over chunk c's rows.  g, y, dy share ld.
int gate_backward(const float* g, const __nv_bfloat16* y, int64_t ld, const float* mods, int64_t ld_mods,
                  const BwdSegs& s, int H, __nv_bfloat16* dy, float* part, cudaStream_t stream);
// Through h = LN(x) (1 + scale) + shift: gx += dx; part[c * 2H + j] = sum dh,
// part[c * 2H + H + j] = sum dh n (n = LN(x)).  x, dh, gx share ld.  With
// aff_w set, through the affine h = LN(x) w + b instead (mods unused; the
// same sums are then the bias and weight gradients' partials).
int ln_modulate_backward(const float* x, const float* dh, float* gx, int64_t ld, const float* mods, int64_t ld_mods,
                         const BwdSegs& s, int H, float* part, cudaStream_t stream, const __nv_bfloat16* aff_w = nullptr);
// Through q = rope(RMSNorm(q_raw) w) for the q (columns [0, H)) and k
// (columns [H, 2H)) gradients in d, in place; rows >= rows_txt are image
// tokens (rotated with the cos / sin table, as the forward epilogue does).
// part[cta * 2d + j] (q scale) and part[cta * 2d + d + j] (k scale): the
// first ctas_txt CTAs cover text rows, the next ctas_img image rows.
struct QkBwdArgs {
    __nv_bfloat16* d; int64_t ldd;
    const __nv_bfloat16* raw; int64_t ldr;
    int rows_txt, rows, heads, head_dim;
    const __nv_bfloat16 *q_scale_txt, *k_scale_txt, *q_scale_img, *k_scale_img;
    const float2* rope_cs;
    int n_img, grid_f, grid_h, grid_w, axes0, axes1, axes2;
    float* part;
    int sets = 2;   // 1: q columns only (a lone query or key block at column 0)
};
int qk_norm_rope_backward(const QkBwdArgs& a, int* ctas_txt, int* ctas_img, cudaStream_t stream);
constexpr int kQkBwdRows = 16;   // rows per CTA of qk_norm_rope_backward
// out[j] = sum over rows of in[r * ld + j] (bf16 or fp32), via ws partials.
size_t colsum_ws_floats(int rows, int ncols);
int colsum(const void* in, bool f32, int64_t ld, int rows, int ncols, float* out, float* ws, cudaStream_t stream);
// B > 0: out[b * ld_out + j] per sample; B == 0: out[j] over every chunk.
int reduce_chunks(const float* part, int64_t ld_part, int ncols, const ChunkSpans& sp, int B, float* out,
                  int64_t ld_out, cudaStream_t stream);
// dx = dy SiLU'(pre) (+ add, fp32 [B, n], when set) (rows < B; fp32 [B, n]) and
// its bf16 copy [rows_pad, n], zero-padded.
int silu_backward(const float* dy, int64_t ld_dy, const __nv_bfloat16* pre, int B, int rows_pad, int n, float* dx,
                  __nv_bfloat16* dxb, cudaStream_t stream, const float* add = nullptr);
// The two products of a Linear applied to B rows (the adaLN modulation and
// the time MLP), HBM-bound kernels in place of the tensor-core GEMM:
//   rows_wgrad  dw[m, n] = sum_b dy[b, m] x[b, n]  (fp32 dy [B, ldy], bf16 x
//               [B, ldx], fp32 dw [M, ldw]; the sum over b in order);
//   rows_dgrad  dx[b, n] = sum_m dy[b, m] w[m, n]  (bf16 w [M, ldw], fp32 dx
//               [B, ldx]; rows_dgrad_chunks(M) fixed chunks of rows, summed in
//               order; B <= 16; part: rows_dgrad_chunks(M) B N floats).
// N, ldx and ldw multiples of 4, 16-byte aligned rows.
constexpr int kRowsDgradMaxChunks = 256;
constexpr int kRowsMaxB = 16;   // batches up to this size use rows_wgrad / rows_dgrad
int rows_wgrad(int B, int M, int N, const float* dy, int64_t ldy, const __nv_bfloat16* x, int64_t ldx, float* dw,
               int64_t ldw, cudaStream_t stream);
int rows_dgrad_chunks(int M);
int rows_dgrad(int B, int M, int N, const float* dy, int64_t ldy, const __nv_bfloat16* w, int64_t ldw, float* dx,
               int64_t ldx, float* part, size_t part_floats, cudaStream_t stream);
// Backward of wan_modulation: from dmods [B, ld] (block l's 6H at l 6H, the
// final layer's shift | scale at L 6H) the bias gradients (blocks.l.mod.b at
// gbias0 + l stride, final.mod.b at gfinal; sums over the batch), d e0 =
// sum over blocks (fp32 [B, 6H] and bf16 [rows_pad, 6H], zero-padded) and
// the final layer's part of d e (fp32 [B, H]).  Fixed summation order.
int wan_modulation_backward(const float* dmods, int64_t ld, int B, int rows_pad, int H, int L, float* gbias0,
                            int64_t stride, float* gfinal, float* de0, __nv_bfloat16* de0b, float* de_fin,
                            cudaStream_t stream);

// mods[b, l*6H + j] = e0[b, j] + bias_l[j] (bias_l = bias0 + l*stride), and
// mods[b, L*6H + j] = e[b, j % H] + fbias[j] for j < 2H (WAN modulation).
int wan_modulation(const float* e, const float* e0, const __nv_bfloat16* bias0, int64_t stride, int L,
                   const __nv_bfloat16* fbias, int B, int H, float* mods, int64_t ld_mods, cudaStream_t stream);

int timestep_embed(const float* t, int B, int dim, __nv_bfloat16* out, cudaStream_t stream);

// ---- the MMDiT forward over caller-chosen buffers (dit.cu) ----------------
// One block's activations: residual before the block, after its attention
// half (double-stream blocks) and after it; LN-modulate outputs h1 / h2;
// normalised and rotated q | k | v; the attention output o (single-stream
// blocks: u holds [o | GELU(mlp)]); the MLP hidden u.  The pre-activation
// copies (raw = QKV or linear1 product + bias, y1 / y2 = gated branches
// before the gate, a1 = MLP1 before GELU) and the attention log-sum-exp are
// written only when set.
struct DitBlockIo {
    float *xin, *xmid, *xout;
    __nv_bfloat16 *h1, *qkv, *raw, *o, *y1, *h2, *a1, *u, *y2;
    float* lse;
    // training only: the attention outputs' low parts (O - bf16(O) in bf16,
    // [R, H] with pitch H; o_lo for the self / joint attention, oc_lo for
    // the WAN cross-attention), so the backward's D = rowsum(dO O) sees O to
    // about 16 bits
    __nv_bfloat16 *o_lo, *oc_lo;
    // WAN blocks (xmid: after the self-attention): the residual after the
    // cross-attention, the affine-LN output, the normalised cross q and text
    // k | v with their raw copies (written only when set), the
    // cross-attention output and its log-sum-exp
    float* x3;
    __nv_bfloat16 *hc, *qc, *qc_raw, *kv, *kv_raw, *oc;
    float* lse_c;
    // training, recompute mode 1: o, o_lo and lse of the self / joint
    // attention already hold this block's values (kept by the first
    // forward), so a re-run of the block skips that attention
    bool attn_kept = false;
};
struct FwdBufs {
    float* mods;
    __nv_bfloat16 *temb, *th, *tc, *pre_fc1, *pre_c, *xb;
    float2* rope;
    float* x0;              // residual after the embeddings
    float* xfin;            // residual after the last block
    __nv_bfloat16* hf;      // final LN-modulate output
    DitBlockIo shared;      // every block's buffers when blocks is null
    const DitBlockIo* blocks;
    DitBlockIo block(int l) const { return blocks ? blocks[l] : shared; }
    // WAN: the timestep embedding e (fp32 [B, H]), the shared modulation e0
    // (fp32 [B, 6H]); the text MLP's pre-GELU copy (when set), its GELU
    // output and the embedded text (bf16 [B N_t, H])
    float *e, *e0;
    __nv_bfloat16 *txt_pre, *txt1, *txth;
    // the attention launches' split scratch (AttnSpec::split_ws), shared by
    // every block: the launches run one after another on the stream
    void* attn_ws = nullptr;
    size_t attn_ws_bytes = 0;
};
int mmdit_forward(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t, float* v_out,
                  const FwdBufs& f, cudaStream_t stream);
// Its four parts: embeddings and modulation; double-stream block l and
// single-stream block l, each from io.xin to io.xout; the final layer.
int mmdit_forward_prologue(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t,
                           const FwdBufs& f, cudaStream_t stream);
int mmdit_forward_double(const ff_dit* m, int B, int l, const DitBlockIo& io, const FwdBufs& f, cudaStream_t stream);
int mmdit_forward_single(const ff_dit* m, int B, int l, const DitBlockIo& io, const FwdBufs& f, cudaStream_t stream);
int mmdit_forward_final(const ff_dit* m, int B, const FwdBufs& f, float* v_out, cudaStream_t stream);
int wan_forward(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t, float* v_out,
                const FwdBufs& f, cudaStream_t stream);
// Its three parts: embeddings and modulation; block l from io.xin to
// io.xout; the final layer from f.xfin.
int wan_forward_prologue(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t,
                         const FwdBufs& f, cudaStream_t stream);
int wan_forward_block(const ff_dit* m, int B, int l, const DitBlockIo& io, const FwdBufs& f, cudaStream_t stream);
int wan_forward_final(const ff_dit* m, int B, const FwdBufs& f, float* v_out, cudaStream_t stream);
// The WAN model's training pass (wan_train.cu): workspace bytes, the forward
// that keeps what the backward reads, and the backward (arguments as
// ff_dit_forward_train / ff_dit_backward, already validated).
size_t wan_train_workspace_bytes(const ff_dit* m, int B);
int wan_forward_train(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t, float* v_out,
                      void* ws, size_t ws_bytes, cudaStream_t stream);
int wan_backward(const ff_dit* m, int B, const void* txt, const float* dv, float* grad, float* dx_t, void* ws,
                 size_t ws_bytes, cudaStream_t stream);
int f32_to_bf16(const float* in, __nv_bfloat16* out, int64_t n, cudaStream_t stream);

}  // namespace ff
