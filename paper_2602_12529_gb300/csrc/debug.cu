// debug.cu -- exported per-kernel entry points (include/ff_debug.h) used by
// the stage-wise parity tests, and the general ff_gemm (include/ff.h).  They
// only marshal arguments to the same launchers ff_dit_velocity uses.
#include "../../include/ff_debug.h"
#include "internal.h"
#include "reduce_jobs.h"

#include <vector>

extern "C" {

int ff_debug_gemm(int M, int N, int K, const void* A, int64_t lda, const void* B, int64_t ldb, const void* bias,
                  int act, int out_f32, void* out, int64_t ldo, cudaStream_t stream) {
    using namespace ff;
    if (act < FF_ACT_NONE || act > FF_ACT_SILU) return set_error(FF_ERR_INVALID_ARG, "bad act %d", act);
    GemmEpilogue e;
    e.act = act;
    e.out_f32 = out_f32 ? 1 : 0;
    e.bias = static_cast<const __nv_bfloat16*>(bias);
    e.out0 = out;
    e.ld0 = ldo;
    return gemm_bf16(A, lda, B, ldb, M, N, K, e, stream);
}

int ff_gemm(int M, int N, int K, const void* A, int64_t lda, int a_layout, const void* B, int64_t ldb, int b_layout,
            const void* bias, int act, int out_f32, void* out, int64_t ldo, cudaStream_t stream) {
    using namespace ff;
    if (act < FF_ACT_NONE || act > FF_ACT_SILU) return set_error(FF_ERR_INVALID_ARG, "gemm: bad act %d", act);
    if ((a_layout != FF_A_MK && a_layout != FF_A_KM) || (b_layout != FF_B_NK && b_layout != FF_B_KN))
        return set_error(FF_ERR_INVALID_ARG, "gemm: bad operand layout (%d, %d)", a_layout, b_layout);
    GemmArgs g{A, lda, B, ldb, M, N, K, GemmEpilogue{}};
    g.a_mn = a_layout == FF_A_KM;
    g.b_mn = b_layout == FF_B_KN;
    g.epi.act = act;
    g.epi.out_f32 = out_f32 ? 1 : 0;
    g.epi.bias = static_cast<const __nv_bfloat16*>(bias);
    g.epi.out0 = out;
    g.epi.ld0 = ldo;
    return gemm_bf16_group(&g, 1, stream);
}

int ff_attention_lse_rows(int n0, int n1) { return ff::attn_lse_rows(n0 < 0 ? 0 : n0, n1 < 0 ? 0 : n1); }

int ff_attention_forward(int B, int heads, int head_dim, int n0, const void* qkv0, int64_t ld0, void* out0,
                         int64_t ldo0, int n1, const void* qkv1, int64_t ld1, void* out1, int64_t ldo1, float* lse,
                         void* ws, size_t ws_bytes, cudaStream_t stream) {
    using namespace ff;
    if (lse && !aligned16(lse)) return set_error(FF_ERR_INVALID_ARG, "attention: lse must be 16-byte aligned");
    if (ws && !aligned16(ws)) return set_error(FF_ERR_INVALID_ARG, "attention: ws must be 16-byte aligned");
    // head h of O lands at columns h d .. h d + d - 1 of its row
    if ((n0 > 0 && ldo0 < static_cast<int64_t>(heads) * head_dim) ||
        (n1 > 0 && ldo1 < static_cast<int64_t>(heads) * head_dim))
        return set_error(FF_ERR_INVALID_ARG, "attention: output pitch below heads * head_dim");
    AttnSpec a;
    const int H = heads * head_dim;
    const void* qkv[2] = {qkv0, qkv1};
    const int64_t ld[2] = {ld0, ld1}, ldo[2] = {ldo0, ldo1};
    void* out[2] = {out0, out1};
    const int n[2] = {n0, n1};
    for (int i = 0; i < 2; ++i) {
        a.q[i] = AttnQuerySeg{static_cast<const __nv_bfloat16*>(qkv[i]), ld[i], n[i],
                              static_cast<__nv_bfloat16*>(out[i]), ldo[i]};
        a.kv[i] = AttnKvSeg{static_cast<const __nv_bfloat16*>(qkv[i]), ld[i], n[i]};
    }
    a.q_col = 0;
    a.k_col = H;
    a.v_col = 2 * H;
    a.B = B;
    a.heads = heads;
    a.head_dim = head_dim;
    a.lse = lse;
    a.split_ws = ws;
    a.split_ws_bytes = ws ? ws_bytes : 0;
    return attention_general(a, stream);
}

int ff_attention_forward_workspace_size(int head_dim, size_t* bytes) {
    using namespace ff;
    if (!bytes) return set_error(FF_ERR_INVALID_ARG, "bytes is null");
    if (head_dim != 64 && head_dim != 128) return set_error(FF_ERR_UNSUPPORTED, "attention: head_dim %d", head_dim);
    *bytes = attention_split_ws_bytes(head_dim);
    return FF_OK;
}

int ff_attention_backward_workspace_size(int B, int heads, int n0, int n1, size_t* bytes) {
    using namespace ff;
    if (!bytes || B <= 0 || heads <= 0 || n0 < 0 || n1 < 0)
        return set_error(FF_ERR_INVALID_ARG, "attention backward: bad workspace query");
    *bytes = attention_backward_ws_bytes(B, heads, n0, n1);
    return FF_OK;
}

int ff_attention_backward(int B, int heads, int head_dim, int n0, const void* qkv0, int64_t ld0, const void* out0,
                          const void* dout0, int64_t ldo0, void* dqkv0, int64_t ldd0, int n1, const void* qkv1,
                          int64_t ld1, const void* out1, const void* dout1, int64_t ldo1, void* dqkv1, int64_t ldd1,
                          const float* lse, void* ws, size_t ws_bytes, cudaStream_t stream) {
    using namespace ff;
    if (lse && !aligned16(lse)) return set_error(FF_ERR_INVALID_ARG, "attention backward: lse must be 16-byte aligned");
    AttnBwdSeg s0{static_cast<const __nv_bfloat16*>(qkv0), ld0, static_cast<const __nv_bfloat16*>(out0),
                  static_cast<const __nv_bfloat16*>(dout0), ldo0, static_cast<__nv_bfloat16*>(dqkv0), ldd0, n0};
    AttnBwdSeg s1{static_cast<const __nv_bfloat16*>(qkv1), ld1, static_cast<const __nv_bfloat16*>(out1),
                  static_cast<const __nv_bfloat16*>(dout1), ldo1, static_cast<__nv_bfloat16*>(dqkv1), ldd1, n1};
    return attention_backward(s0, s1, B, heads, head_dim, lse, ws, ws_bytes, stream);
}

int ff_cross_attention_forward(int B, int heads, int head_dim, int nq, const void* q, int64_t ldq, int nk,
                               const void* kv, int64_t ldkv, void* out, int64_t ldo, float* lse, cudaStream_t stream) {
    using namespace ff;
    if (nq <= 0 || nk <= 0) return set_error(FF_ERR_INVALID_ARG, "cross-attention: nq and nk must be positive");
    if (lse && !aligned16(lse)) return set_error(FF_ERR_INVALID_ARG, "cross-attention: lse must be 16-byte aligned");
    if (ldo < static_cast<int64_t>(heads) * head_dim)
        return set_error(FF_ERR_INVALID_ARG, "cross-attention: output pitch below heads * head_dim");
    AttnSpec a;
    a.q[0] = AttnQuerySeg{static_cast<const __nv_bfloat16*>(q), ldq, nq, static_cast<__nv_bfloat16*>(out), ldo};
    a.q[1] = AttnQuerySeg{nullptr, 0, 0, nullptr, 0};
    a.kv[0] = AttnKvSeg{static_cast<const __nv_bfloat16*>(kv), ldkv, nk};
    a.kv[1] = AttnKvSeg{nullptr, 0, 0};
    a.q_col = 0;
    a.k_col = 0;
    a.v_col = heads * head_dim;
    a.B = B;
    a.heads = heads;
    a.head_dim = head_dim;
    a.lse = lse;
    return attention_general(a, stream);
}

int ff_cross_attention_backward(int B, int heads, int head_dim, int nq, const void* q, int64_t ldq, const void* out,
                                const void* dout, int64_t ldo, void* dq, int64_t lddq, int nk, const void* kv,
                                int64_t ldkv, void* dkv, int64_t lddkv, const float* lse, void* ws, size_t ws_bytes,
                                cudaStream_t stream) {
    using namespace ff;
    if (nq <= 0 || nk <= 0) return set_error(FF_ERR_INVALID_ARG, "cross-attention: nq and nk must be positive");
    if (lse && !aligned16(lse)) return set_error(FF_ERR_INVALID_ARG, "cross-attention: lse must be 16-byte aligned");
    const int64_t H = static_cast<int64_t>(heads) * head_dim;
    if (lddkv < 2 * H) return set_error(FF_ERR_INVALID_ARG, "cross-attention: lddkv %lld < 2H", (long long)lddkv);
    auto* g = static_cast<__nv_bfloat16*>(dkv);
    AttnBwdSpec a{};
    a.q[0] = AttnBwdQuerySeg{static_cast<const __nv_bfloat16*>(q), ldq, nq, static_cast<const __nv_bfloat16*>(out), ldo,
                             static_cast<const __nv_bfloat16*>(dout), ldo, static_cast<__nv_bfloat16*>(dq), lddq};
    a.kv[0] = AttnBwdKvSeg{static_cast<const __nv_bfloat16*>(kv), ldkv, nk, g, g ? g + H : nullptr, lddkv};
    a.q_col = 0;
    a.k_col = 0;
    a.v_col = static_cast<int>(H);
    a.B = B;
    a.heads = heads;
    a.head_dim = head_dim;
    a.lse = lse;
    return attention_backward_general(a, ws, ws_bytes, stream);
}

int ff_debug_gemm_gated(int M, int N, int K, const void* A, int64_t lda, const void* B, int64_t ldb, const void* bias,
                        float* resid, int64_t ld_resid, const float* gate, int64_t ld_gate, int rows_per_sample,
                        cudaStream_t stream) {
    using namespace ff;
    GemmEpilogue e;
    e.epi = EPI_GATED_RESIDUAL;
    e.bias = static_cast<const __nv_bfloat16*>(bias);
    e.resid = resid;
    e.ld_resid = ld_resid;
    e.gate = gate;
    e.ld_gate = ld_gate;
    e.rows_per_sample = rows_per_sample;
    return gemm_bf16(A, lda, B, ldb, M, N, K, e, stream);
}

int ff_debug_attention(int B, int heads, int head_dim, int n0, const void* qkv0, int64_t ld0, void* out0,
                       int64_t ldo0, int n1, const void* qkv1, int64_t ld1, void* out1, int64_t ldo1,
                       cudaStream_t stream) {
    using namespace ff;
    if ((n0 > 0 && ldo0 < static_cast<int64_t>(heads) * head_dim) ||
        (n1 > 0 && ldo1 < static_cast<int64_t>(heads) * head_dim))
        return set_error(FF_ERR_INVALID_ARG, "attention: output pitch below heads * head_dim");
    AttnSegment s0{static_cast<const __nv_bfloat16*>(qkv0), ld0, static_cast<__nv_bfloat16*>(out0), ldo0, n0};
    AttnSegment s1{static_cast<const __nv_bfloat16*>(qkv1), ld1, static_cast<__nv_bfloat16*>(out1), ldo1, n1};
    return attention(s0, s1, B, heads, head_dim, heads * head_dim, stream);
}

int ff_debug_attention_launch(int mode) {
    using namespace ff;
    if (mode < 0 || mode > 3) return set_error(FF_ERR_INVALID_ARG, "attention launch mode %d (0 to 3)", mode);
    return attention_launch_override(mode);
}

int ff_debug_ln_modulate(int rows, int H, const float* x, const float* mods, int64_t ld_mods, int shift_off,
                         int scale_off, int tokens_per_sample, void* out, cudaStream_t stream) {
    using namespace ff;
    if (!x || !mods || !out || rows < 0 || H <= 0 || tokens_per_sample <= 0)
        return set_error(FF_ERR_INVALID_ARG, "ln_modulate: bad arguments");
    LnModArgs a{};
    a.x = x; a.ldx = H; a.out = static_cast<__nv_bfloat16*>(out); a.ldo = H; a.rows = rows; a.H = H;
    a.rows_txt = 0; a.n_txt = 1; a.n_img = tokens_per_sample; a.mods = mods; a.ld_mods = ld_mods;
    a.shift_txt = a.shift_img = shift_off;
    a.scale_txt = a.scale_img = scale_off;
    return ln_modulate(a, stream);
}

int ff_debug_qk_norm_rope(int rows, int rows_txt, int heads, int head_dim, void* qkv, int64_t ld, const void* q_scale,
                          const void* k_scale, int grid_f, int grid_h, int grid_w, const int* rope_axes,
                          float rope_theta, cudaStream_t stream) {
    using namespace ff;
    if (!qkv || !q_scale || !k_scale || !rope_axes || rows < 0 || rows_txt < 0 || rows_txt > rows)
        return set_error(FF_ERR_INVALID_ARG, "qk_norm_rope: bad arguments");
    if (rope_axes[0] + rope_axes[1] + rope_axes[2] != head_dim)
        return set_error(FF_ERR_INVALID_ARG, "qk_norm_rope: rope_axes must sum to head_dim");
    QkNormRopeArgs a{};
    a.qkv = static_cast<__nv_bfloat16*>(qkv); a.ld = ld; a.rows = rows; a.heads = heads; a.head_dim = head_dim;
    a.rows_txt = rows_txt; a.n_img = grid_f * grid_h * grid_w; a.grid_f = grid_f; a.grid_h = grid_h; a.grid_w = grid_w;
    a.axes0 = rope_axes[0]; a.axes1 = rope_axes[1]; a.axes2 = rope_axes[2]; a.theta = rope_theta;
    a.q_scale_txt = a.q_scale_img = static_cast<const __nv_bfloat16*>(q_scale);
    a.k_scale_txt = a.k_scale_img = static_cast<const __nv_bfloat16*>(k_scale);
    a.col[0] = 0;
    a.col[1] = heads * head_dim;
    a.rope = 1;
    return qk_norm_rope(a, stream);
}

int ff_debug_reduce_chunks(int n, int B, const float* part, float* out, const int64_t* part_off,
                           const int64_t* ld_part, const int* ncols, const int* first, const int* count,
                           const int* per_sample, const int64_t* out_off, const int64_t* ld_out, cudaStream_t stream) {
    using namespace ff;
    if (n < 0 || B < 0) return set_error(FF_ERR_INVALID_ARG, "reduce_chunks: n=%d B=%d", n, B);
    if (n == 0) return FF_OK;
    if (!part || !out || !part_off || !ld_part || !ncols || !first || !count || !per_sample || !out_off || !ld_out)
        return set_error(FF_ERR_INVALID_ARG, "reduce_chunks: null argument");
    std::vector<ReduceJob> jobs(n);
    for (int i = 0; i < n; ++i) {
        if (first[2 * i] < 0 || count[2 * i] <= 0 || count[2 * i + 1] < 0 || (count[2 * i + 1] > 0 && first[2 * i + 1] < 0) ||
            part_off[i] < 0 || out_off[i] < 0 || ld_part[i] < ncols[i] || (per_sample[i] && ld_out[i] < ncols[i]))
            return set_error(FF_ERR_INVALID_ARG, "reduce_chunks: job %d has a bad span or pitch", i);
        ChunkSpans sp{};
        sp.n = count[2 * i + 1] > 0 ? 2 : 1;
        for (int k = 0; k < sp.n; ++k) {
            sp.first[k] = first[2 * i + k];
            sp.count[k] = count[2 * i + k];
        }
        jobs[i] = ReduceJob{part + part_off[i], ld_part[i], ncols[i], sp, per_sample[i] ? 1 : 0, out + out_off[i],
                            ld_out[i]};
    }
    return reduce_chunks_batch(jobs.data(), n, B, stream);
}

}  // extern "C"
