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
    // EPI_GATED_RESIDUAL: resid[m, n] += gate[(m / rows_per_sample) * ld_gate + n] * (acc + bias)
    float* resid = nullptr;
    int64_t ld_resid = 0;
    const float* gate = nullptr;
    int64_t ld_gate = 0;
    int rows_per_sample = 1;
};

int gemm_bf16(const void* A, int64_t lda, const void* B, int64_t ldb, int M, int N, int K,
              const GemmEpilogue& epi, cudaStream_t stream);

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
};
int ln_modulate(const LnModArgs& a, cudaStream_t stream);

// In-place per-head RMSNorm of q and k plus RoPE on a bf16 qkv buffer
// [rows, ld] with q at column 0, k at column H.
struct QkNormRopeArgs {
    __nv_bfloat16* qkv; int64_t ld;
    int rows, heads, head_dim;
    int rows_txt, n_img;               // rows >= rows_txt are image tokens
    int grid_f, grid_h, grid_w;
    int axes0, axes1, axes2;
    float theta;
    const __nv_bfloat16* q_scale_txt; const __nv_bfloat16* k_scale_txt;
    const __nv_bfloat16* q_scale_img; const __nv_bfloat16* k_scale_img;
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

int timestep_embed(const float* t, int B, int dim, __nv_bfloat16* out, cudaStream_t stream);
int f32_to_bf16(const float* in, __nv_bfloat16* out, int64_t n, cudaStream_t stream);

}  // namespace ff
