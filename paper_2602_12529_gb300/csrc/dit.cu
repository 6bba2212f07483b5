// dit.cu -- the DiT velocity entry points: weight-blob layout, model handle,
// workspace plan, and the launch sequence of one velocity call.
//
// Activation layout in the workspace (R_t = B N_t text rows, R_i = B N_i
// image rows, R = R_t + R_i): every per-token buffer is "stream-major" --
// rows [0, R_t) are the text tokens of samples 0..B-1 (sample-major), rows
// [R_t, R) the image tokens.  A double-stream block runs each stream's GEMMs
// on its contiguous row range with its own weights; a single-stream block
// runs one GEMM over all R rows (row order is irrelevant to a Linear); only
// attention (segments per sample) and the adaLN vectors (sample per row) need
// the split.
//
//   mods  fp32 [B, W_mod]      all adaLN vectors (one GEMM per call)
//   x     fp32 [R, H]          residual stream
//   h     bf16 [R, H]          LN-modulated GEMM operand
//   qkv   bf16 [R, 3H]         q | k | v (q, k RMSNorm'd and rotated by the QKV GEMM epilogue)
//   o     bf16 [R, H]          attention output (double-stream blocks)
//   u     bf16 [R, H + F]      MLP hidden [R, F] (double) or [attn | GELU(mlp)] (single)
#include <string.h>

#include <string>
#include <unordered_map>
#include <vector>

#include "internal.h"

struct ff_dit {
    ff_dit_config cfg;
    const __nv_bfloat16* w;
    std::unordered_map<std::string, int64_t> off;
    int64_t mod_width;
    // training pass: 0 keeps every activation; 1 keeps the block inputs and
    // the attention outputs, re-running the rest of each block before its
    // backward; 2 keeps the block inputs only
    int train_recompute = 0;
    int attn_split = 1;   // attention launches may split their last round (ff_dit_set_attention_split)
    mutable int fwd_recompute = -1;   // the mode of the latest ff_dit_forward_train (-1: none yet)
};

namespace ff {
namespace {

struct Spec {
    std::string name;
    int ndim;
    int64_t s0, s1;
};

int64_t mod_width(const ff_dit_config& c) {
    const int64_t H = c.hidden;
    return c.n_double * 12 * H + c.n_single * 3 * H + 2 * H;
}

// Same order and names as the oracle's parameter list.
std::vector<Spec> specs(const ff_dit_config& c) {
    const int64_t H = c.hidden, F = c.mlp, P = c.patch_dim, d = c.head_dim;
    std::vector<Spec> s;
    auto mat = [&](const std::string& n, int64_t o, int64_t i) { s.push_back({n, 2, o, i}); };
    auto vec = [&](const std::string& n, int64_t o) { s.push_back({n, 1, o, 0}); };
    mat("t_embed.fc1.w", H, c.time_freq_dim); vec("t_embed.fc1.b", H);
    mat("t_embed.fc2.w", H, H); vec("t_embed.fc2.b", H);
    mat("mod.w", mod_width(c), H); vec("mod.b", mod_width(c));
    mat("img_in.w", H, P); vec("img_in.b", H);
    mat("txt_in.w", H, c.txt_dim); vec("txt_in.b", H);
    for (int l = 0; l < c.n_double; ++l) {
        for (const char* st : {"img", "txt"}) {
            const std::string p = "double." + std::to_string(l) + "." + st + ".";
            mat(p + "qkv.w", 3 * H, H); vec(p + "qkv.b", 3 * H);
            vec(p + "q_norm.scale", d); vec(p + "k_norm.scale", d);
            mat(p + "proj.w", H, H); vec(p + "proj.b", H);
            mat(p + "mlp1.w", F, H); vec(p + "mlp1.b", F);
            mat(p + "mlp2.w", H, F); vec(p + "mlp2.b", H);
        }
    }
    for (int l = 0; l < c.n_single; ++l) {
        const std::string p = "single." + std::to_string(l) + ".";
        mat(p + "linear1.w", 3 * H + F, H); vec(p + "linear1.b", 3 * H + F);
        vec(p + "q_norm.scale", d); vec(p + "k_norm.scale", d);
        mat(p + "linear2.w", H, H + F); vec(p + "linear2.b", H);
    }
    mat("final.w", P, H); vec("final.b", P);
    return s;
}

// WAN-style DiT parameters, same order and names as the oracle's list.
std::vector<Spec> specs_wan(const ff_dit_config& c) {
    const int64_t H = c.hidden, F = c.mlp, P = c.patch_dim, d = c.head_dim;
    std::vector<Spec> s;
    auto mat = [&](const std::string& n, int64_t o, int64_t i) { s.push_back({n, 2, o, i}); };
    auto vec = [&](const std::string& n, int64_t o) { s.push_back({n, 1, o, 0}); };
    mat("t_embed.fc1.w", H, c.time_freq_dim); vec("t_embed.fc1.b", H);
    mat("t_embed.fc2.w", H, H); vec("t_embed.fc2.b", H);
    mat("mod.w", 6 * H, H); vec("mod.b", 6 * H);
    mat("img_in.w", H, P); vec("img_in.b", H);
    mat("txt_in.w", H, c.txt_dim); vec("txt_in.b", H);
    mat("txt_in2.w", H, H); vec("txt_in2.b", H);
    for (int l = 0; l < c.n_double; ++l) {
        const std::string p = "blocks." + std::to_string(l) + ".";
        vec(p + "mod.b", 6 * H);
        mat(p + "qkv.w", 3 * H, H); vec(p + "qkv.b", 3 * H);
        vec(p + "q_norm.scale", d); vec(p + "k_norm.scale", d);
        mat(p + "proj.w", H, H); vec(p + "proj.b", H);
        vec(p + "cross_norm.scale", H); vec(p + "cross_norm.b", H);
        mat(p + "cross_q.w", H, H); vec(p + "cross_q.b", H); vec(p + "cross_q_norm.scale", d);
        mat(p + "cross_kv.w", 2 * H, H); vec(p + "cross_kv.b", 2 * H); vec(p + "cross_k_norm.scale", d);
        mat(p + "cross_proj.w", H, H); vec(p + "cross_proj.b", H);
        mat(p + "mlp1.w", F, H); vec(p + "mlp1.b", F);
        mat(p + "mlp2.w", H, F); vec(p + "mlp2.b", H);
    }
    vec("final.mod.b", 2 * H);
    mat("final.w", P, H); vec("final.b", P);
    return s;
}

std::vector<Spec> specs_for(const ff_dit_config& c) { return c.arch == FF_ARCH_WAN ? specs_wan(c) : specs(c); }

int validate(const ff_dit_config* c) {
    if (!c) return set_error(FF_ERR_INVALID_ARG, "config is null");
    if (c->arch != FF_ARCH_MMDIT && c->arch != FF_ARCH_WAN) return set_error(FF_ERR_UNSUPPORTED, "arch %d not supported", c->arch);
    if (c->arch == FF_ARCH_WAN && (c->n_single != 0 || c->n_double < 1))
        return set_error(FF_ERR_INVALID_ARG, "WAN: n_double = blocks >= 1, n_single = 0");
    if (c->hidden <= 0 || c->hidden % 128) return set_error(FF_ERR_UNSUPPORTED, "hidden %d must be a multiple of 128", c->hidden);
    if (c->head_dim != 64 && c->head_dim != 128) return set_error(FF_ERR_UNSUPPORTED, "head_dim %d", c->head_dim);
    if (c->heads * c->head_dim != c->hidden) return set_error(FF_ERR_INVALID_ARG, "heads * head_dim != hidden");
    if (c->mlp <= 0 || c->mlp % 64) return set_error(FF_ERR_UNSUPPORTED, "mlp %d must be a multiple of 64", c->mlp);
    if (c->n_double < 0 || c->n_single < 0 || c->n_double + c->n_single < 1)
        return set_error(FF_ERR_INVALID_ARG, "need at least one block");
    if (c->patch_dim <= 0 || c->patch_dim % 32) return set_error(FF_ERR_UNSUPPORTED, "patch_dim %d", c->patch_dim);
    if (c->txt_dim <= 0 || c->txt_dim % 8) return set_error(FF_ERR_UNSUPPORTED, "txt_dim %d", c->txt_dim);
    if (c->n_txt <= 0) return set_error(FF_ERR_UNSUPPORTED, "n_txt must be positive");
    if (c->grid_f <= 0 || c->grid_h <= 0 || c->grid_w <= 0) return set_error(FF_ERR_INVALID_ARG, "bad latent grid");
    if (c->rope_axes[0] % 2 || c->rope_axes[1] % 2 || c->rope_axes[2] % 2 || c->rope_axes[0] < 0 ||
        c->rope_axes[1] < 0 || c->rope_axes[2] < 0 ||
        c->rope_axes[0] + c->rope_axes[1] + c->rope_axes[2] != c->head_dim)
        return set_error(FF_ERR_INVALID_ARG, "rope_axes must be even and sum to head_dim");
    if (!(c->rope_theta > 1.0f)) return set_error(FF_ERR_INVALID_ARG, "rope_theta must be > 1");
    if (c->time_freq_dim <= 0 || c->time_freq_dim % 64) return set_error(FF_ERR_UNSUPPORTED, "time_freq_dim %d", c->time_freq_dim);
    return FF_OK;
}

constexpr size_t kAlign = 256;
size_t up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

struct Workspace {
    float* mods;
    __nv_bfloat16 *temb, *th, *tc;
    float* x;
    __nv_bfloat16 *xb, *h, *qkv, *o, *u;
    // WAN only
    float *e, *e0;
    __nv_bfloat16 *txt1, *txth, *kvc;
    float2* rope;   // cos / sin table of every rotation angle
    void* attn_ws;  // the attention launches' split scratch
    size_t bytes;
};

Workspace plan(const ff_dit_config& c, int B, uint8_t* base) {
    const size_t H = c.hidden, F = c.mlp;
    const size_t Ni = static_cast<size_t>(c.grid_f) * c.grid_h * c.grid_w;
    const bool wan = c.arch == FF_ARCH_WAN;
    // WAN keeps only latent tokens in the residual stream; text lives in its own buffers
    const size_t R = static_cast<size_t>(B) * (wan ? Ni : c.n_txt + Ni);
    const size_t Rt = static_cast<size_t>(B) * c.n_txt;
    const size_t Wm = wan ? static_cast<size_t>(c.n_double) * 6 * H + 2 * H : static_cast<size_t>(mod_width(c));
    size_t o = 0;
    Workspace w{};
    auto take = [&](size_t bytes) { uint8_t* p = base ? base + o : nullptr; o += up(bytes); return p; };
    w.mods = reinterpret_cast<float*>(take(static_cast<size_t>(B) * Wm * 4));
    w.temb = reinterpret_cast<__nv_bfloat16*>(take(static_cast<size_t>(B) * c.time_freq_dim * 2));
    w.th = reinterpret_cast<__nv_bfloat16*>(take(B * H * 2));
    w.tc = reinterpret_cast<__nv_bfloat16*>(take(B * H * 2));
    w.x = reinterpret_cast<float*>(take(R * H * 4));
    w.xb = reinterpret_cast<__nv_bfloat16*>(take(B * Ni * c.patch_dim * 2));
    w.h = reinterpret_cast<__nv_bfloat16*>(take(R * H * 2));
    w.qkv = reinterpret_cast<__nv_bfloat16*>(take(R * 3 * H * 2));
    w.o = reinterpret_cast<__nv_bfloat16*>(take(R * H * 2));
    w.u = reinterpret_cast<__nv_bfloat16*>(take(R * (H + F) * 2));
    w.rope = reinterpret_cast<float2*>(take(static_cast<size_t>(rope_table_size(
        c.grid_f, c.grid_h, c.grid_w, c.rope_axes[0], c.rope_axes[1], c.rope_axes[2])) * sizeof(float2)));
    w.attn_ws = take(attention_split_ws_bytes(c.head_dim));
    if (wan) {
        w.e = reinterpret_cast<float*>(take(B * H * 4));
        w.e0 = reinterpret_cast<float*>(take(B * 6 * H * 4));
        w.txt1 = reinterpret_cast<__nv_bfloat16*>(take(Rt * H * 2));
        w.txth = reinterpret_cast<__nv_bfloat16*>(take(Rt * H * 2));
        w.kvc = reinterpret_cast<__nv_bfloat16*>(take(Rt * 2 * H * 2));
    }
    w.bytes = o;
    return w;
}

// Fused per-head RMSNorm (+ RoPE when table is set) of the q | k columns.
void set_qk_norm(GemmEpilogue& e, const ff_dit_config& c, int qk_cols, const __nv_bfloat16* qs,
                 const __nv_bfloat16* ks, const float2* table, int rope_row0) {
    e.qk_cols = qk_cols;
    e.head_dim = c.head_dim;
    e.q_scale = qs;
    e.k_scale = ks;
    e.rope_cs = table;
    e.rope_row0 = rope_row0;
    e.n_img = c.grid_f * c.grid_h * c.grid_w;
    e.grid_f = c.grid_f;
    e.grid_h = c.grid_h;
    e.grid_w = c.grid_w;
    e.axes0 = c.rope_axes[0];
    e.axes1 = c.rope_axes[1];
    e.axes2 = c.rope_axes[2];
}


}  // namespace

// WAN-style velocity: latent tokens only in the residual stream; the text is
// embedded once per call and feeds every block's cross-attention keys and
// values.  Buffers come from f as for mmdit_forward (one shared set for the
// inference call, one set per block with the raw copies for training).  In
// three parts, so a training pass can re-run one block alone:
//   wan_forward_prologue  rotation table, timestep embedding, modulation,
//                         patch and text embeddings (into f.x0, f.txth);
//   wan_forward_block     block l from io.xin to io.xout;
//   wan_forward_final     the final layer from f.xfin to v.
int wan_forward_prologue(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t,
                         const FwdBufs& f, cudaStream_t stream) {
    const ff_dit_config& c = m->cfg;
    const int H = c.hidden, P = c.patch_dim, L = c.n_double;
    const int Nt = c.n_txt, Ni = c.grid_f * c.grid_h * c.grid_w;
    const int Rt = B * Nt, Ri = B * Ni;
    const int64_t Wm = m->mod_width;
    auto W = [&](const std::string& n) { return m->w + m->off.at(n); };

    // rotation table; timestep embedding e (fp32), SiLU(e) (bf16), e0 = SiLU(e) W_mod^T + b; per-block modulation
    FF_TRY(rope_table(f.rope, c.grid_f, c.grid_h, c.grid_w, c.rope_axes[0], c.rope_axes[1], c.rope_axes[2],
                      c.rope_theta, stream));
    FF_TRY(timestep_embed(t, B, c.time_freq_dim, f.temb, stream));
    {
        GemmEpilogue e;
        e.rows_gemv = 1; e.act = ACT_SILU; e.bias = W("t_embed.fc1.b"); e.out0 = f.th; e.ld0 = H;
        e.aux = f.pre_fc1; e.ld_aux = H;
        FF_TRY(gemm_bf16(f.temb, c.time_freq_dim, W("t_embed.fc1.w"), c.time_freq_dim, B, H, c.time_freq_dim, e, stream));
    }
    {
        GemmEpilogue e;
        e.rows_gemv = 1; e.out_f32 = 1; e.bias = W("t_embed.fc2.b"); e.out0 = f.e; e.ld0 = H;
        FF_TRY(gemm_bf16(f.th, H, W("t_embed.fc2.w"), H, B, H, H, e, stream));
    }
    {
        GemmEpilogue e;
        e.rows_gemv = 1; e.act = ACT_SILU; e.bias = W("t_embed.fc2.b"); e.out0 = f.tc; e.ld0 = H;
        e.aux = f.pre_c; e.ld_aux = H;
        FF_TRY(gemm_bf16(f.th, H, W("t_embed.fc2.w"), H, B, H, H, e, stream));
    }
    {
        GemmEpilogue e;
        e.rows_gemv = 1; e.out_f32 = 1; e.bias = W("mod.b"); e.out0 = f.e0; e.ld0 = 6 * H;
        FF_TRY(gemm_bf16(f.tc, H, W("mod.w"), H, B, 6 * H, H, e, stream));
    }
    const int64_t stride = L > 1 ? m->off.at("blocks.1.mod.b") - m->off.at("blocks.0.mod.b") : 0;
    FF_TRY(wan_modulation(f.e, f.e0, W("blocks.0.mod.b"), stride, L, W("final.mod.b"), B, H, f.mods, Wm, stream));

    // latent tokens and text embeddings
    FF_TRY(f32_to_bf16(x_t, f.xb, static_cast<int64_t>(Ri) * P, stream));
    {
        GemmEpilogue e;
        e.out_f32 = 1; e.bias = W("img_in.b"); e.out0 = f.x0; e.ld0 = H;
        FF_TRY(gemm_bf16(f.xb, P, W("img_in.w"), P, Ri, H, P, e, stream));
    }
    {
        GemmEpilogue e;
        e.act = ACT_GELU; e.bias = W("txt_in.b"); e.out0 = f.txt1; e.ld0 = H;
        e.aux = f.txt_pre; e.ld_aux = H;
        FF_TRY(gemm_bf16(txt, c.txt_dim, W("txt_in.w"), c.txt_dim, Rt, H, c.txt_dim, e, stream));
    }
    {
        GemmEpilogue e;
        e.bias = W("txt_in2.b"); e.out0 = f.txth; e.ld0 = H;
        FF_TRY(gemm_bf16(f.txt1, H, W("txt_in2.w"), H, Rt, H, H, e, stream));
    }
    return FF_OK;
}

namespace {
LnModArgs wan_ln_args(const ff_dit* m, int B, const FwdBufs& f) {
    const ff_dit_config& c = m->cfg;
    const int H = c.hidden, Ni = c.grid_f * c.grid_h * c.grid_w;
    LnModArgs la{};
    la.ldx = H; la.ldo = H; la.rows = B * Ni; la.H = H;
    la.rows_txt = 0; la.n_txt = 1; la.n_img = Ni; la.mods = f.mods; la.ld_mods = m->mod_width;
    return la;
}
}  // namespace

int wan_forward_block(const ff_dit* m, int B, int l, const DitBlockIo& io, const FwdBufs& f, cudaStream_t stream) {
    const ff_dit_config& c = m->cfg;
    const int H = c.hidden, F = c.mlp, d = c.head_dim;
    const int Nt = c.n_txt, Ni = c.grid_f * c.grid_h * c.grid_w;
    const int Rt = B * Nt, Ri = B * Ni;
    const int64_t Wm = m->mod_width;
    auto W = [&](const std::string& n) { return m->w + m->off.at(n); };
    LnModArgs la = wan_ln_args(m, B, f);
    {
        const std::string p = "blocks." + std::to_string(l) + ".";
        const int base = l * 6 * H;
        // self-attention
        la.x = io.xin; la.out = io.h1;
        la.aff_w = la.aff_b = nullptr;
        la.shift_txt = la.shift_img = base;
        la.scale_txt = la.scale_img = base + H;
        FF_TRY(ln_modulate(la, stream));
        {
            GemmEpilogue e;
            e.bias = W(p + "qkv.b"); e.out0 = io.qkv; e.ld0 = 3 * H;
            e.aux = io.raw; e.ld_aux = 3 * H;
            set_qk_norm(e, c, 2 * H, W(p + "q_norm.scale"), W(p + "k_norm.scale"), f.rope, 0);
            FF_TRY(gemm_bf16(io.h1, H, W(p + "qkv.w"), H, Ri, 3 * H, H, e, stream));
        }
        if (!io.attn_kept) {   // a re-run in recompute mode 1 finds O, its low part and lse kept
            AttnSpec a{};
            a.q[0] = AttnQuerySeg{nullptr, 0, 0, nullptr, 0};
            a.q[1] = AttnQuerySeg{io.qkv, 3 * H, Ni, io.o, H, io.o_lo, H};
            a.kv[0] = AttnKvSeg{nullptr, 0, 0};
            a.kv[1] = AttnKvSeg{io.qkv, 3 * H, Ni};
            a.q_col = 0; a.k_col = H; a.v_col = 2 * H;
            a.B = B; a.heads = c.heads; a.head_dim = d;
            a.lse = io.lse;
            a.split_ws = f.attn_ws; a.split_ws_bytes = f.attn_ws_bytes;
            FF_TRY(attention_general(a, stream));
        }
        {
            GemmEpilogue e;
            e.epi = EPI_GATED_RESIDUAL; e.bias = W(p + "proj.b");
            e.resid = io.xin; e.ld_resid = H;
            if (io.xmid != io.xin) e.resid_out = io.xmid;
            e.gate = f.mods + base + 2 * H; e.ld_gate = Wm; e.rows_per_sample = Ni;
            e.aux = io.y1; e.ld_aux = H;
            FF_TRY(gemm_bf16(io.o, H, W(p + "proj.w"), H, Ri, H, H, e, stream));
        }
        // cross-attention to the text
        la.x = io.xmid; la.out = io.hc;
        la.aff_w = W(p + "cross_norm.scale");
        la.aff_b = W(p + "cross_norm.b");
        FF_TRY(ln_modulate(la, stream));
        {
            GemmEpilogue e;   // cross q with its RMSNorm fused (no rotation)
            e.bias = W(p + "cross_q.b"); e.out0 = io.qc; e.ld0 = H;
            e.aux = io.qc_raw; e.ld_aux = H;
            set_qk_norm(e, c, H, W(p + "cross_q_norm.scale"), W(p + "cross_q_norm.scale"), nullptr, 0);
            FF_TRY(gemm_bf16(io.hc, H, W(p + "cross_q.w"), H, Ri, H, H, e, stream));
        }
        {
            GemmEpilogue e;   // cross k | v of the text, RMSNorm on k fused
            e.bias = W(p + "cross_kv.b"); e.out0 = io.kv; e.ld0 = 2 * H;
            e.aux = io.kv_raw; e.ld_aux = 2 * H;
            set_qk_norm(e, c, H, W(p + "cross_k_norm.scale"), W(p + "cross_k_norm.scale"), nullptr, 0);
            FF_TRY(gemm_bf16(f.txth, H, W(p + "cross_kv.w"), H, Rt, 2 * H, H, e, stream));
        }
        {
            AttnSpec a{};
            a.q[0] = AttnQuerySeg{nullptr, 0, 0, nullptr, 0};
            a.q[1] = AttnQuerySeg{io.qc, H, Ni, io.oc, H, io.oc_lo, H};
            a.kv[0] = AttnKvSeg{io.kv, 2 * H, Nt};
            a.kv[1] = AttnKvSeg{nullptr, 0, 0};
            a.q_col = 0; a.k_col = 0; a.v_col = H;
            a.B = B; a.heads = c.heads; a.head_dim = d;
            a.lse = io.lse_c;
            a.split_ws = f.attn_ws; a.split_ws_bytes = f.attn_ws_bytes;
            FF_TRY(attention_general(a, stream));
        }
        {
            GemmEpilogue e;   // plain residual: no gate on the cross-attention branch
            e.epi = EPI_GATED_RESIDUAL; e.bias = W(p + "cross_proj.b");
            e.resid = io.xmid; e.ld_resid = H; e.gate = nullptr; e.rows_per_sample = Ni;
            if (io.x3 != io.xmid) e.resid_out = io.x3;
            FF_TRY(gemm_bf16(io.oc, H, W(p + "cross_proj.w"), H, Ri, H, H, e, stream));
        }
        // FFN
        la.x = io.x3; la.out = io.h2;
        la.aff_w = la.aff_b = nullptr;
        la.shift_txt = la.shift_img = base + 3 * H;
        la.scale_txt = la.scale_img = base + 4 * H;
        FF_TRY(ln_modulate(la, stream));
        {
            GemmEpilogue e;
            e.act = ACT_GELU; e.bias = W(p + "mlp1.b"); e.out0 = io.u; e.ld0 = F;
            e.aux = io.a1; e.ld_aux = F;
            FF_TRY(gemm_bf16(io.h2, H, W(p + "mlp1.w"), H, Ri, F, H, e, stream));
        }
        {
            GemmEpilogue e;
            e.epi = EPI_GATED_RESIDUAL; e.bias = W(p + "mlp2.b");
            e.resid = io.x3; e.ld_resid = H;
            if (io.xout != io.x3) e.resid_out = io.xout;
            e.gate = f.mods + base + 5 * H; e.ld_gate = Wm; e.rows_per_sample = Ni;
            e.aux = io.y2; e.ld_aux = H;
            FF_TRY(gemm_bf16(io.u, F, W(p + "mlp2.w"), F, Ri, H, F, e, stream));
        }
    }
    return FF_OK;
}

int wan_forward_final(const ff_dit* m, int B, const FwdBufs& f, float* v_out, cudaStream_t stream) {
    const ff_dit_config& c = m->cfg;
    const int H = c.hidden, P = c.patch_dim, L = c.n_double;
    const int Ni = c.grid_f * c.grid_h * c.grid_w;
    const int Ri = B * Ni;
    auto W = [&](const std::string& n) { return m->w + m->off.at(n); };
    LnModArgs la = wan_ln_args(m, B, f);
    la.x = f.xfin; la.out = f.hf;
    la.aff_w = la.aff_b = nullptr;
    la.shift_txt = la.shift_img = L * 6 * H;
    la.scale_txt = la.scale_img = L * 6 * H + H;
    FF_TRY(ln_modulate(la, stream));
    GemmEpilogue e;
    e.out_f32 = 1; e.bias = W("final.b"); e.out0 = v_out; e.ld0 = P;
    return gemm_bf16(f.hf, H, W("final.w"), H, Ri, P, H, e, stream);
}

int wan_forward(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t, float* v_out,
                const FwdBufs& f, cudaStream_t stream) {
    FF_TRY(wan_forward_prologue(m, B, x_t, txt, t, f, stream));
    for (int l = 0; l < m->cfg.n_double; ++l) FF_TRY(wan_forward_block(m, B, l, f.block(l), f, stream));
    return wan_forward_final(m, B, f, v_out, stream);
}

// The MMDiT velocity: timestep MLP and every adaLN vector, embeddings, the
// double- and single-stream blocks, the final layer.  Buffers come from f:
// the inference call passes one shared set (residual updated in place), the
// training forward one set per block with the pre-activation copies the
// backward reads.  In four parts, so a training pass can re-run one block:
// prologue (rotation table, time MLP, modulation, embeddings into f.x0),
// double-stream block l, single-stream block l (io.xin -> io.xout), final.
int mmdit_forward_prologue(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t,
                           const FwdBufs& f, cudaStream_t stream) {
    const ff_dit_config& c = m->cfg;
    const int H = c.hidden, P = c.patch_dim;
    const int Nt = c.n_txt, Ni = c.grid_f * c.grid_h * c.grid_w;
    const int Rt = B * Nt, Ri = B * Ni;
    const int64_t Wm = m->mod_width;
    auto W = [&](const std::string& n) { return m->w + m->off.at(n); };

    // ---- rotation table, timestep embedding MLP and every adaLN vector
    FF_TRY(rope_table(f.rope, c.grid_f, c.grid_h, c.grid_w, c.rope_axes[0], c.rope_axes[1], c.rope_axes[2],
                      c.rope_theta, stream));
    FF_TRY(timestep_embed(t, B, c.time_freq_dim, f.temb, stream));
    {
        GemmEpilogue e;
        e.rows_gemv = 1; e.act = ACT_SILU; e.bias = W("t_embed.fc1.b"); e.out0 = f.th; e.ld0 = H;
        e.aux = f.pre_fc1; e.ld_aux = H;
        FF_TRY(gemm_bf16(f.temb, c.time_freq_dim, W("t_embed.fc1.w"), c.time_freq_dim, B, H, c.time_freq_dim, e, stream));
    }
    {
        GemmEpilogue e;   // SiLU(c): only the modulation GEMM consumes c
        e.rows_gemv = 1; e.act = ACT_SILU; e.bias = W("t_embed.fc2.b"); e.out0 = f.tc; e.ld0 = H;
        e.aux = f.pre_c; e.ld_aux = H;
        FF_TRY(gemm_bf16(f.th, H, W("t_embed.fc2.w"), H, B, H, H, e, stream));
    }
    {
        GemmEpilogue e;
        e.rows_gemv = 1; e.out_f32 = 1; e.bias = W("mod.b"); e.out0 = f.mods; e.ld0 = Wm;
        FF_TRY(gemm_bf16(f.tc, H, W("mod.w"), H, B, static_cast<int>(Wm), H, e, stream));
    }

    // ---- patch and text embeddings into the residual stream
    FF_TRY(f32_to_bf16(x_t, f.xb, static_cast<int64_t>(Ri) * P, stream));
    {
        // the long-K text product first, so its few expensive tiles start at
        // once and the short patch-embedding tiles fill in behind them
        GemmArgs g[2];
        g[0] = GemmArgs{txt, c.txt_dim, W("txt_in.w"), c.txt_dim, Rt, H, c.txt_dim, GemmEpilogue{}};
        g[0].epi.out_f32 = 1; g[0].epi.bias = W("txt_in.b"); g[0].epi.out0 = f.x0; g[0].epi.ld0 = H;
        g[1] = GemmArgs{f.xb, P, W("img_in.w"), P, Ri, H, P, GemmEpilogue{}};
        g[1].epi.out_f32 = 1; g[1].epi.bias = W("img_in.b"); g[1].epi.out0 = f.x0 + static_cast<int64_t>(Rt) * H;
        g[1].epi.ld0 = H;
        FF_TRY(gemm_bf16_group(g, 2, stream));
    }
    return FF_OK;
}

namespace {
LnModArgs mmdit_ln_args(const ff_dit* m, int B, const FwdBufs& f) {
    const ff_dit_config& c = m->cfg;
    const int Nt = c.n_txt, Ni = c.grid_f * c.grid_h * c.grid_w;
    LnModArgs la{};
    la.ldx = c.hidden; la.ldo = c.hidden; la.rows = B * (Nt + Ni); la.H = c.hidden;
    la.rows_txt = B * Nt; la.n_txt = Nt; la.n_img = Ni; la.mods = f.mods; la.ld_mods = m->mod_width;
    return la;
}
struct Stream { const char* name; int row0, rows, tokens; int64_t mod; };
}  // namespace

int mmdit_forward_double(const ff_dit* m, int B, int l, const DitBlockIo& io, const FwdBufs& f,
                         cudaStream_t stream) {
    const ff_dit_config& c = m->cfg;
    const int H = c.hidden, F = c.mlp;
    const int Nt = c.n_txt, Ni = c.grid_f * c.grid_h * c.grid_w;
    const int Rt = B * Nt, Ri = B * Ni;
    const int64_t Wm = m->mod_width;
    auto W = [&](const std::string& n) { return m->w + m->off.at(n); };
    auto rows = [](auto* p, int64_t r, int64_t ld) { return p ? p + r * ld : p; };
    LnModArgs la = mmdit_ln_args(m, B, f);
    {
        const int64_t base = static_cast<int64_t>(l) * 12 * H;
        const Stream st[2] = {{"txt", 0, Rt, Nt, base + 6 * H}, {"img", Rt, Ri, Ni, base}};
        const std::string pre = "double." + std::to_string(l) + ".";
        // LN-modulate 1
        la.x = io.xin; la.out = io.h1;
        la.shift_txt = static_cast<int>(st[0].mod); la.scale_txt = static_cast<int>(st[0].mod + H);
        la.shift_img = static_cast<int>(st[1].mod); la.scale_img = static_cast<int>(st[1].mod + H);
        FF_TRY(ln_modulate(la, stream));
        // Each GEMM below runs both streams in one launch: image problem
        // first, the (smaller) text problem filling its tail.
        const Stream* ord[2] = {&st[1], &st[0]};
        // QKV, with q / k RMSNorm and RoPE fused into the epilogue
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i) {
                const Stream& s = *ord[i];
                const std::string p = pre + s.name + ".";
                g[i] = GemmArgs{io.h1 + static_cast<int64_t>(s.row0) * H, H, W(p + "qkv.w"), H, s.rows, 3 * H, H,
                                GemmEpilogue{}};
                GemmEpilogue& e = g[i].epi;
                e.bias = W(p + "qkv.b"); e.out0 = io.qkv + static_cast<int64_t>(s.row0) * 3 * H; e.ld0 = 3 * H;
                e.aux = rows(io.raw, s.row0, 3 * H); e.ld_aux = 3 * H;
                set_qk_norm(e, c, 2 * H, W(p + "q_norm.scale"), W(p + "k_norm.scale"), s.row0 ? f.rope : nullptr, 0);
            }
            FF_TRY(gemm_bf16_group(g, 2, stream));
        }
        if (!io.attn_kept) {   // a re-run in recompute mode 1 finds O, its low part and lse kept
            AttnSegment a0{io.qkv, 3 * H, io.o, H, Nt, io.o_lo, H};
            AttnSegment a1{io.qkv + static_cast<int64_t>(Rt) * 3 * H, 3 * H, io.o + static_cast<int64_t>(Rt) * H, H, Ni,
                           io.o_lo ? io.o_lo + static_cast<int64_t>(Rt) * H : nullptr, H};
            FF_TRY(attention(a0, a1, B, c.heads, c.head_dim, H, stream, io.lse, f.attn_ws, f.attn_ws_bytes));
        }
        // projection + gated residual (gate1)
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i) {
                const Stream& s = *ord[i];
                const std::string p = pre + s.name + ".";
                g[i] = GemmArgs{io.o + static_cast<int64_t>(s.row0) * H, H, W(p + "proj.w"), H, s.rows, H, H,
                                GemmEpilogue{}};
                GemmEpilogue& e = g[i].epi;
                e.epi = EPI_GATED_RESIDUAL; e.bias = W(p + "proj.b");
                e.resid = io.xin + static_cast<int64_t>(s.row0) * H; e.ld_resid = H;
                if (io.xmid != io.xin) e.resid_out = io.xmid + static_cast<int64_t>(s.row0) * H;
                e.gate = f.mods + s.mod + 2 * H; e.ld_gate = Wm; e.rows_per_sample = s.tokens;
                e.aux = rows(io.y1, s.row0, H); e.ld_aux = H;
            }
            FF_TRY(gemm_bf16_group(g, 2, stream));
        }
        // LN-modulate 2
        la.x = io.xmid; la.out = io.h2;
        la.shift_txt = static_cast<int>(st[0].mod + 3 * H); la.scale_txt = static_cast<int>(st[0].mod + 4 * H);
        la.shift_img = static_cast<int>(st[1].mod + 3 * H); la.scale_img = static_cast<int>(st[1].mod + 4 * H);
        FF_TRY(ln_modulate(la, stream));
        // MLP
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i) {
                const Stream& s = *ord[i];
                const std::string p = pre + s.name + ".";
                g[i] = GemmArgs{io.h2 + static_cast<int64_t>(s.row0) * H, H, W(p + "mlp1.w"), H, s.rows, F, H,
                                GemmEpilogue{}};
                GemmEpilogue& e = g[i].epi;
                e.act = ACT_GELU; e.bias = W(p + "mlp1.b"); e.out0 = io.u + static_cast<int64_t>(s.row0) * F; e.ld0 = F;
                e.aux = rows(io.a1, s.row0, F); e.ld_aux = F;
            }
            FF_TRY(gemm_bf16_group(g, 2, stream));
        }
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i) {
                const Stream& s = *ord[i];
                const std::string p = pre + s.name + ".";
                g[i] = GemmArgs{io.u + static_cast<int64_t>(s.row0) * F, F, W(p + "mlp2.w"), F, s.rows, H, F,
                                GemmEpilogue{}};
                GemmEpilogue& e = g[i].epi;
                e.epi = EPI_GATED_RESIDUAL; e.bias = W(p + "mlp2.b");
                e.resid = io.xmid + static_cast<int64_t>(s.row0) * H; e.ld_resid = H;
                if (io.xout != io.xmid) e.resid_out = io.xout + static_cast<int64_t>(s.row0) * H;
                e.gate = f.mods + s.mod + 5 * H; e.ld_gate = Wm; e.rows_per_sample = s.tokens;
                e.aux = rows(io.y2, s.row0, H); e.ld_aux = H;
            }
            FF_TRY(gemm_bf16_group(g, 2, stream));
        }
    }
    return FF_OK;
}

int mmdit_forward_single(const ff_dit* m, int B, int l, const DitBlockIo& io, const FwdBufs& f,
                         cudaStream_t stream) {
    const ff_dit_config& c = m->cfg;
    const int H = c.hidden, F = c.mlp;
    const int Nt = c.n_txt, Ni = c.grid_f * c.grid_h * c.grid_w;
    const int Rt = B * Nt, Ri = B * Ni, R = Rt + Ri;
    const int64_t Wm = m->mod_width;
    auto W = [&](const std::string& n) { return m->w + m->off.at(n); };
    auto rows = [](auto* p, int64_t r, int64_t ld) { return p ? p + r * ld : p; };
    LnModArgs la = mmdit_ln_args(m, B, f);
    {
        const int64_t off = static_cast<int64_t>(c.n_double) * 12 * H + static_cast<int64_t>(l) * 3 * H;
        const std::string p = "single." + std::to_string(l) + ".";
        la.x = io.xin; la.out = io.h1;
        la.shift_txt = la.shift_img = static_cast<int>(off);
        la.scale_txt = la.scale_img = static_cast<int>(off + H);
        FF_TRY(ln_modulate(la, stream));
        {
            GemmEpilogue e;   // [q k v] -> qkv ; GELU(mlp) -> u[:, H:]
            e.bias = W(p + "linear1.b");
            e.out0 = io.qkv; e.ld0 = 3 * H;
            e.split_n = 3 * H; e.out1 = io.u; e.ld1 = H + F; e.col1 = H;
            e.act = ACT_GELU; e.act_from = 3 * H;
            e.aux = io.raw; e.ld_aux = 3 * H + F;
            set_qk_norm(e, c, 2 * H, W(p + "q_norm.scale"), W(p + "k_norm.scale"), f.rope, Rt);
            FF_TRY(gemm_bf16(io.h1, H, W(p + "linear1.w"), H, R, 3 * H + F, H, e, stream));
        }
        {
            AttnSegment a0{io.qkv, 3 * H, io.u, H + F, Nt, io.o_lo, H};
            AttnSegment a1{io.qkv + static_cast<int64_t>(Rt) * 3 * H, 3 * H, io.u + static_cast<int64_t>(Rt) * (H + F),
                           H + F, Ni, io.o_lo ? io.o_lo + static_cast<int64_t>(Rt) * H : nullptr, H};
            FF_TRY(attention(a0, a1, B, c.heads, c.head_dim, H, stream, io.lse, f.attn_ws, f.attn_ws_bytes));
        }
        // linear2 + gated residual: one launch, the two segments as two
        // problems (the sample index of a row differs per segment)
        {
            const Stream st[2] = {{"img", Rt, Ri, Ni, off}, {"txt", 0, Rt, Nt, off}};
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i) {
                const Stream& s = st[i];
                g[i] = GemmArgs{io.u + static_cast<int64_t>(s.row0) * (H + F), H + F, W(p + "linear2.w"), H + F,
                                s.rows, H, H + F, GemmEpilogue{}};
                GemmEpilogue& e = g[i].epi;
                e.epi = EPI_GATED_RESIDUAL; e.bias = W(p + "linear2.b");
                e.resid = io.xin + static_cast<int64_t>(s.row0) * H; e.ld_resid = H;
                if (io.xout != io.xin) e.resid_out = io.xout + static_cast<int64_t>(s.row0) * H;
                e.gate = f.mods + off + 2 * H; e.ld_gate = Wm; e.rows_per_sample = s.tokens;
                e.aux = rows(io.y2, s.row0, H); e.ld_aux = H;
            }
            FF_TRY(gemm_bf16_group(g, 2, stream));
        }
    }
    return FF_OK;
}

int mmdit_forward_final(const ff_dit* m, int B, const FwdBufs& f, float* v_out, cudaStream_t stream) {
    const ff_dit_config& c = m->cfg;
    const int H = c.hidden, P = c.patch_dim;
    const int Nt = c.n_txt, Ni = c.grid_f * c.grid_h * c.grid_w;
    const int Rt = B * Nt, Ri = B * Ni;
    auto W = [&](const std::string& n) { return m->w + m->off.at(n); };
    LnModArgs la = mmdit_ln_args(m, B, f);
    // ---- final layer on image tokens -> v (fp32)
    {
        const int64_t off = static_cast<int64_t>(c.n_double) * 12 * H + static_cast<int64_t>(c.n_single) * 3 * H;
        LnModArgs fl = la;
        fl.x = f.xfin + static_cast<int64_t>(Rt) * H; fl.rows = Ri; fl.rows_txt = 0; fl.out = f.hf;
        fl.shift_img = fl.shift_txt = static_cast<int>(off);
        fl.scale_img = fl.scale_txt = static_cast<int>(off + H);
        FF_TRY(ln_modulate(fl, stream));
        GemmEpilogue e;
        e.out_f32 = 1; e.bias = W("final.b"); e.out0 = v_out; e.ld0 = P;
        FF_TRY(gemm_bf16(f.hf, H, W("final.w"), H, Ri, P, H, e, stream));
    }
    return FF_OK;
}

int mmdit_forward(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t, float* v_out,
                  const FwdBufs& f, cudaStream_t stream) {
    FF_TRY(mmdit_forward_prologue(m, B, x_t, txt, t, f, stream));
    for (int l = 0; l < m->cfg.n_double; ++l) FF_TRY(mmdit_forward_double(m, B, l, f.block(l), f, stream));
    for (int l = 0; l < m->cfg.n_single; ++l)
        FF_TRY(mmdit_forward_single(m, B, l, f.block(m->cfg.n_double + l), f, stream));
    return mmdit_forward_final(m, B, f, v_out, stream);
}

const ff_dit_config& model_config(const ff_dit* m) { return m->cfg; }
const __nv_bfloat16* model_weights(const ff_dit* m) { return m->w; }
int64_t model_offset(const ff_dit* m, const char* name) {
    const auto it = m->off.find(name);
    return it == m->off.end() ? -1 : it->second;
}
int64_t model_mod_width(const ff_dit* m) { return m->mod_width; }
int model_train_recompute(const ff_dit* m) { return m->train_recompute; }
int model_attention_split(const ff_dit* m) { return m->attn_split; }
void model_note_forward_train(const ff_dit* m) { m->fwd_recompute = m->train_recompute; }
int model_forward_train_mode(const ff_dit* m) { return m->fwd_recompute; }

}  // namespace ff

extern "C" {

int ff_dit_weight_layout(const ff_dit_config* cfg, ff_tensor_desc* out, int capacity, int* count,
                         int64_t* total_elems) {
    using namespace ff;
    FF_TRY(validate(cfg));
    if (!count || !total_elems) return set_error(FF_ERR_INVALID_ARG, "count/total_elems is null");
    const std::vector<Spec> s = specs_for(*cfg);
    int64_t off = 0;
    for (size_t i = 0; i < s.size(); ++i) {
        const int64_t n = s[i].ndim == 2 ? s[i].s0 * s[i].s1 : s[i].s0;
        if (out && static_cast<int>(i) < capacity) {
            memset(&out[i], 0, sizeof(ff_tensor_desc));
            strncpy(out[i].name, s[i].name.c_str(), sizeof(out[i].name) - 1);
            out[i].offset = off;
            out[i].ndim = s[i].ndim;
            out[i].shape[0] = s[i].s0;
            out[i].shape[1] = s[i].ndim == 2 ? s[i].s1 : 0;
        }
        off += (n + 63) / 64 * 64;   // every tensor starts on a 128-byte boundary
    }
    *count = static_cast<int>(s.size());
    *total_elems = off;
    return FF_OK;
}

int ff_dit_create(const ff_dit_config* cfg, const void* weights_dev, ff_dit** out) {
    using namespace ff;
    FF_TRY(validate(cfg));
    if (!weights_dev || !out) return set_error(FF_ERR_INVALID_ARG, "weights/out is null");
    if (!aligned16(weights_dev)) return set_error(FF_ERR_INVALID_ARG, "weight blob must be 16-byte aligned");
    ff_dit* m = new ff_dit();
    m->cfg = *cfg;
    m->w = static_cast<const __nv_bfloat16*>(weights_dev);
    m->mod_width = cfg->arch == FF_ARCH_WAN ? static_cast<int64_t>(cfg->n_double) * 6 * cfg->hidden + 2 * cfg->hidden
                                            : mod_width(*cfg);
    int64_t off = 0;
    for (const Spec& s : specs_for(*cfg)) {
        m->off[s.name] = off;
        const int64_t n = s.ndim == 2 ? s.s0 * s.s1 : s.s0;
        off += (n + 63) / 64 * 64;
    }
    *out = m;
    return FF_OK;
}

int ff_dit_destroy(ff_dit* m) {
    delete m;
    return FF_OK;
}

int ff_dit_set_train_recompute(ff_dit* m, int on) {
    using namespace ff;
    if (!m) return set_error(FF_ERR_INVALID_ARG, "model is null");
    if (on < 0 || on > 2) return set_error(FF_ERR_INVALID_ARG, "recompute mode %d (0, 1 or 2)", on);
    m->train_recompute = on;
    return FF_OK;
}

int ff_dit_set_attention_split(ff_dit* m, int on) {
    using namespace ff;
    if (!m) return set_error(FF_ERR_INVALID_ARG, "model is null");
    if (on != 0 && on != 1) return set_error(FF_ERR_INVALID_ARG, "attention split %d (0 or 1)", on);
    m->attn_split = on;
    return FF_OK;
}

int ff_dit_workspace_size(const ff_dit* m, int B, size_t* bytes) {
    using namespace ff;
    if (!m || !bytes) return set_error(FF_ERR_INVALID_ARG, "model/bytes is null");
    if (B <= 0) return set_error(FF_ERR_INVALID_ARG, "B=%d must be positive", B);
    *bytes = plan(m->cfg, B, nullptr).bytes;
    return FF_OK;
}

int ff_dit_velocity(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t, float* v_out, void* ws,
                    size_t ws_bytes, cudaStream_t stream) {
    using namespace ff;
    if (!m) return set_error(FF_ERR_INVALID_ARG, "model is null");
    if (B <= 0) return set_error(FF_ERR_INVALID_ARG, "B=%d must be positive", B);
    if (!x_t || !txt || !t || !v_out || !ws) return set_error(FF_ERR_INVALID_ARG, "null pointer argument");
    if (!aligned16(x_t) || !aligned16(txt) || !aligned16(v_out) || (reinterpret_cast<uintptr_t>(ws) % kAlign))
        return set_error(FF_ERR_INVALID_ARG, "misaligned pointer (arrays 16 B, workspace 256 B)");
    const ff_dit_config& c = m->cfg;
    const Workspace w = plan(c, B, static_cast<uint8_t*>(ws));
    if (ws_bytes < w.bytes) return set_error(FF_ERR_WORKSPACE, "workspace %zu B < %zu B needed", ws_bytes, w.bytes);

    FwdBufs f{};
    f.mods = w.mods; f.temb = w.temb; f.th = w.th; f.tc = w.tc; f.xb = w.xb; f.rope = w.rope;
    f.x0 = f.xfin = w.x;
    f.hf = w.h;
    f.attn_ws = m->attn_split ? w.attn_ws : nullptr;
    f.attn_ws_bytes = attention_split_ws_bytes(c.head_dim);
    f.shared = DitBlockIo{w.x, w.x, w.x, w.h, w.qkv, nullptr, w.o, nullptr, w.h, nullptr, w.u, nullptr, nullptr};
    if (c.arch == FF_ARCH_WAN) {
        // one buffer per role, reused by every block: the residual in place,
        // cross q in the QKV buffer, the cross-attention output in o
        f.shared.x3 = w.x;
        f.shared.hc = w.h;
        f.shared.qc = w.qkv;
        f.shared.kv = w.kvc;
        f.shared.oc = w.o;
        f.e = w.e; f.e0 = w.e0; f.txt1 = w.txt1; f.txth = w.txth;
        return wan_forward(m, B, x_t, txt, t, v_out, f, stream);
    }
    return mmdit_forward(m, B, x_t, txt, t, v_out, f, stream);
}

}  // extern "C"
