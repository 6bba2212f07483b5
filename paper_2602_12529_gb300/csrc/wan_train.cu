// wan_train.cu -- the training pass of the WAN-style velocity (the forward
// every GRPO-style trainer runs "again for training", Sec. 1, and its
// gradient), behind the same entries as the MMDiT's (ff_dit_forward_train,
// ff_dit_backward).
//
// Per block, in reverse: the gated FFN half, the ungated cross-attention half
// (affine LayerNorm; latent queries, text keys / values; every block adds its
// k | v input gradient into the embedded text's gradient), the gated
// self-attention half.  Then the patch embedding, the text MLP, and the
// shared modulation e0 + b_l / e + b_final back through SiLU(e) and the
// timestep MLP.  Products run on the tcgen05 GEMM (weight gradients with both
// operands MN-major, input gradients with W MN-major), the attention
// backward on attention_backward_general, the rest on backward.cu's row
// kernels; every sum over tokens or samples has a fixed order, so the
// gradient is deterministic.
//
// Workspace (written by the forward, read by the backward; R_i = B N_i latent
// rows, R_t = B N_t text rows):
//   mods fp32 [B, W_mod]; e fp32 [B, H], e0 fp32 [B, 6H]; time-MLP operands
//   (bf16, zero-padded to a multiple of 8 rows) and their pre-activation
//   copies; the text MLP's pre-GELU copy, GELU output and result [R_t, H];
//   per block: x_in, x_mid, x_3 fp32 [R_i, H]; h1, o, y1, hc, q_c (+ raw),
//   oc, h2, y2 bf16 [R_i, H]; raw and normalised qkv [R_i, 3H]; k | v of the
//   text (+ raw) [R_t, 2H]; a1, u [R_i, F]; both attentions' log-sum-exp;
//   the final residual and LN-modulate output; then the backward's scratch.
// In recompute mode (ff_dit_set_train_recompute) the blocks share one set of
// those activations and only their input residuals are kept, with (mode 1)
// each block's self-attention output, its low part and lse; the backward
// re-runs block l's forward (bit-identical, every kernel is deterministic)
// just before its backward, skipping the self-attention in mode 1.
#include <initializer_list>
#include <string>
#include <vector>

#include "internal.h"
#include "reduce_jobs.h"

namespace ff {
namespace {

constexpr size_t kAlign = 256;
size_t up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

struct WanPlan {
    FwdBufs f;
    std::vector<DitBlockIo> blk;
    int rows_pad;
    // backward scratch
    float *gx, *dh, *part, *cs_ws, *dtxt;
    __nv_bfloat16 *dy, *dbig, *dob, *dkv, *dyt, *dvb;
    void* attn_ws;
    size_t attn_ws_bytes;
    float *dmods, *de0, *de_fin, *dtc, *dc, *dth, *da;
    float* rows_part;          // rows_dgrad's partial sums
    size_t rows_part_floats;
    __nv_bfloat16 *de0_b, *dc_b, *da_b;
    size_t bytes;
};

WanPlan plan(const ff_dit_config& c, int64_t Wm, int B, uint8_t* base, int recompute) {
    const size_t H = c.hidden, F = c.mlp, P = c.patch_dim, tf = c.time_freq_dim, d = c.head_dim;
    const size_t Nt = c.n_txt, Ni = static_cast<size_t>(c.grid_f) * c.grid_h * c.grid_w;
    const size_t Rt = B * Nt, Ri = B * Ni;
    const size_t Kp = (B + 7) / 8 * 8;
    size_t o = 0;
    auto take = [&](size_t bytes) { uint8_t* p = base ? base + o : nullptr; o += up(bytes); return p; };
    auto f32 = [&](size_t n) { return reinterpret_cast<float*>(take(n * 4)); };
    auto b16 = [&](size_t n) { return reinterpret_cast<__nv_bfloat16*>(take(n * 2)); };
    WanPlan p{};
    p.rows_pad = static_cast<int>(Kp);
    FwdBufs& f = p.f;
    f.mods = f32(B * Wm);
    f.e = f32(B * H);
    f.e0 = f32(B * 6 * H);
    f.temb = b16(Kp * tf);
    f.th = b16(Kp * H);
    f.tc = b16(Kp * H);
    f.pre_fc1 = b16(B * H);
    f.pre_c = b16(B * H);
    f.xb = b16(Ri * P);
    f.txt_pre = b16(Rt * H);
    f.txt1 = b16(Rt * H);
    f.txth = b16(Rt * H);
    f.rope = reinterpret_cast<float2*>(take(static_cast<size_t>(rope_table_size(
        c.grid_f, c.grid_h, c.grid_w, c.rope_axes[0], c.rope_axes[1], c.rope_axes[2])) * sizeof(float2)));
    f.attn_ws_bytes = attention_split_ws_bytes(c.head_dim);
    f.attn_ws = take(f.attn_ws_bytes);
    const int L = c.n_double;
    const size_t lse_n = static_cast<size_t>(B) * c.heads * attn_lse_rows(0, static_cast<int>(Ni));
    p.blk.resize(L);
    float* x = f32(Ri * H);
    f.x0 = x;
    // recompute: one activation set shared by every block (re-filled by the
    // backward); kept per block: the input and, in mode 1, the
    // self-attention's O, its low part and lse
    DitBlockIo shared{};
    for (int l = 0; l < L; ++l) {
        DitBlockIo& io = p.blk[l];
        if (recompute && l > 0) {
            io = shared;
            io.xin = x;
            if (recompute == 1) {
                io.o = b16(Ri * H);
                io.o_lo = b16(Ri * H);
                io.lse = f32(lse_n);
            }
            x = f32(Ri * H);
            io.xout = x;
            continue;
        }
        io = DitBlockIo{};
        io.xin = x;
        io.h1 = b16(Ri * H);
        io.raw = b16(Ri * 3 * H);
        io.qkv = b16(Ri * 3 * H);
        io.lse = f32(lse_n);
        io.o = b16(Ri * H);
        io.o_lo = b16(Ri * H);
        io.y1 = b16(Ri * H);
        io.xmid = f32(Ri * H);
        io.hc = b16(Ri * H);
        io.qc_raw = b16(Ri * H);
        io.qc = b16(Ri * H);
        io.kv_raw = b16(Rt * 2 * H);
        io.kv = b16(Rt * 2 * H);
        io.oc = b16(Ri * H);
        io.oc_lo = b16(Ri * H);
        io.lse_c = f32(lse_n);
        io.x3 = f32(Ri * H);
        io.h2 = b16(Ri * H);
        io.a1 = b16(Ri * F);
        io.u = b16(Ri * F);
        io.y2 = b16(Ri * H);
        x = f32(Ri * H);
        io.xout = x;
        shared = io;
    }
    f.xfin = x;
    f.hf = b16(Ri * H);
    f.blocks = nullptr;   // set by the caller once the plan has its final address

    const size_t wide = std::max(F, 3 * H);
    p.gx = f32(Ri * H);
    p.dh = f32(Ri * H);
    p.dtxt = f32(Rt * H);
    p.dy = b16(Ri * H);
    p.dbig = b16(Ri * wide);
    p.dob = b16(Ri * H);
    p.dkv = b16(Rt * 2 * H);
    p.dyt = b16(Rt * H);
    p.dvb = b16(Ri * P);
    const size_t chunks = static_cast<size_t>(B) * bwd_chunks(static_cast<int>(Ni));
    const size_t qk_ctas = std::max((Ri + kQkBwdRows - 1) / kQkBwdRows, (Rt + kQkBwdRows - 1) / kQkBwdRows);
    p.part = f32(std::max(chunks * 2 * H, qk_ctas * 2 * d));
    size_t cs = colsum_ws_floats(static_cast<int>(Ri), static_cast<int>(std::max(wide, P)));
    cs = std::max(cs, colsum_ws_floats(static_cast<int>(Rt), static_cast<int>(2 * H)));
    cs = std::max(cs, colsum_ws_floats(B, static_cast<int>(6 * H)));
    p.cs_ws = f32(cs);
    p.attn_ws_bytes = attention_backward_ws_bytes(B, c.heads, 0, static_cast<int>(Ni));
    p.attn_ws = take(p.attn_ws_bytes);
    p.dmods = f32(B * Wm);
    p.de0 = f32(B * 6 * H);
    p.de0_b = b16(Kp * 6 * H);
    p.de_fin = f32(B * H);
    p.dtc = f32(Kp * H);
    p.dc = f32(B * H);
    p.dc_b = b16(Kp * H);
    p.dth = f32(Kp * H);
    p.da = f32(B * H);
    p.da_b = b16(Kp * H);
    p.rows_part_floats = B <= kRowsMaxB ? static_cast<size_t>(rows_dgrad_chunks(static_cast<int>(6 * H))) * B * H : 0;
    p.rows_part = f32(p.rows_part_floats);
    p.bytes = o;
    return p;
}

}  // namespace

size_t wan_train_workspace_bytes(const ff_dit* m, int B) {
    return plan(model_config(m), model_mod_width(m), B, nullptr, model_train_recompute(m)).bytes;
}

int wan_forward_train(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t, float* v_out,
                      void* ws, size_t ws_bytes, cudaStream_t stream) {
    const ff_dit_config& c = model_config(m);
    WanPlan p = plan(c, model_mod_width(m), B, static_cast<uint8_t*>(ws), model_train_recompute(m));
    if (!model_attention_split(m)) p.f.attn_ws = nullptr;
    if (ws_bytes < p.bytes) return set_error(FF_ERR_WORKSPACE, "workspace %zu B < %zu B needed", ws_bytes, p.bytes);
    p.f.blocks = p.blk.data();
    // the time-MLP operands' padding rows (the weight-gradient products read them)
    if (p.rows_pad > B) {
        const size_t pad = static_cast<size_t>(p.rows_pad - B);
        if (cudaMemsetAsync(p.f.temb + static_cast<size_t>(B) * c.time_freq_dim, 0, pad * c.time_freq_dim * 2, stream) ||
            cudaMemsetAsync(p.f.th + static_cast<size_t>(B) * c.hidden, 0, pad * c.hidden * 2, stream) ||
            cudaMemsetAsync(p.f.tc + static_cast<size_t>(B) * c.hidden, 0, pad * c.hidden * 2, stream))
            return set_error(FF_ERR_CUDA, "forward_train: memset failed");
    }
    return wan_forward(m, B, x_t, txt, t, v_out, p.f, stream);
}

int wan_backward(const ff_dit* m, int B, const void* txt, const float* dv, float* grad, float* dx_t, void* ws,
                 size_t ws_bytes, cudaStream_t stream) {
    const ff_dit_config& c = model_config(m);
    const int64_t Wm = model_mod_width(m);
    const int recompute = model_train_recompute(m);
    WanPlan p = plan(c, Wm, B, static_cast<uint8_t*>(ws), recompute);
    if (!model_attention_split(m)) p.f.attn_ws = nullptr;
    if (ws_bytes < p.bytes) return set_error(FF_ERR_WORKSPACE, "workspace %zu B < %zu B needed", ws_bytes, p.bytes);
    const FwdBufs& f = p.f;
    const int H = c.hidden, F = c.mlp, P = c.patch_dim, d = c.head_dim, heads = c.heads, tf = c.time_freq_dim;
    const int L = c.n_double;
    const int Nt = c.n_txt, Ni = c.grid_f * c.grid_h * c.grid_w;
    const int Rt = B * Nt, Ri = B * Ni;
    const int Kp = p.rows_pad;
    const int cps = bwd_chunks(Ni);
    const int W3 = 3 * H;
    const __nv_bfloat16* w0 = model_weights(m);
    auto W = [&](const std::string& n) { return w0 + model_offset(m, n.c_str()); };
    auto G = [&](const std::string& n) { return grad + model_offset(m, n.c_str()); };
    auto gemm1 = [&](GemmArgs g) { return gemm_bf16_group(&g, 1, stream); };
    const BwdSeg img{0, Ni, 0, 0};
    // per-sample sums of the chunk partials (columns [col, col + H) of part) into dmods
    auto per_sample = [&](int col, float* out) {
        return ReduceJob{p.part + col, 2 * H, H, chunk_span(0, cps), 1, out, Wm};
    };
    // sums over every chunk (ncols columns of part at col, pitch ld)
    auto total = [&](int count, int col, int64_t ld, int ncols, float* out) {
        return ReduceJob{p.part + col, ld, ncols, chunk_span(0, count), 0, out, 0};
    };
    // the sums that follow one backward kernel, in one launch
    auto reduce = [&](std::initializer_list<ReduceJob> jobs) {
        return reduce_chunks_batch(jobs.begin(), static_cast<int>(jobs.size()), B, stream);
    };
    auto gate = [&](const __nv_bfloat16* y, int col_gate, float* dgate, float* dbias) {
        BwdSeg sg = img;
        sg.col_a = col_gate;
        const BwdSegs s = bwd_segs(&sg, 1, B);
        FF_TRY(gate_backward(p.gx, y, H, f.mods, Wm, s, H, p.dy, p.part, stream));
        return reduce({per_sample(0, dgate), total(B * cps, H, 2 * H, H, dbias)});
    };
    auto lnmod = [&](const float* x, int col_shift) {
        BwdSeg sg = img;
        sg.col_b = col_shift + H;
        const BwdSegs s = bwd_segs(&sg, 1, B);
        FF_TRY(ln_modulate_backward(x, p.dh, p.gx, H, f.mods, Wm, s, H, p.part, stream));
        return reduce({per_sample(0, p.dmods + col_shift), per_sample(H, p.dmods + col_shift + H)});
    };

    // ---- final layer: v = LNmod(x) W_f^T + b_f (shift | scale at L 6H)
    const int off_f = L * 6 * H;
    FF_TRY(f32_to_bf16(dv, p.dvb, static_cast<int64_t>(Ri) * P, stream));
    FF_TRY(gemm1(gemm_wgrad(p.dvb, P, f.hf, H, P, H, Ri, G("final.w"))));
    FF_TRY(colsum(dv, true, P, Ri, P, G("final.b"), p.cs_ws, stream));
    {
        GemmArgs g = gemm_dgrad(p.dvb, P, W("final.w"), Ri, H, P);
        g.epi.out_f32 = 1; g.epi.out0 = p.dh; g.epi.ld0 = H;
        FF_TRY(gemm1(g));
    }
    if (cudaMemsetAsync(p.gx, 0, static_cast<size_t>(Ri) * H * 4, stream) != cudaSuccess ||
        cudaMemsetAsync(p.dtxt, 0, static_cast<size_t>(Rt) * H * 4, stream) != cudaSuccess)
        return set_error(FF_ERR_CUDA, "backward: memset failed");
    FF_TRY(lnmod(f.xfin, off_f));

    // ---- blocks, last first
    for (int l = L - 1; l >= 0; --l) {
        const DitBlockIo& io = p.blk[l];
        // recompute: this block's activations again, from its kept input
        if (recompute) {
            DitBlockIo r = io;
            r.attn_kept = recompute == 1;   // mode 1: the self-attention's outputs were kept
            FF_TRY(wan_forward_block(m, B, l, r, f, stream));
        }
        const int base = l * 6 * H;
        const std::string pre = "blocks." + std::to_string(l) + ".";
        // FFN half: x_out = x3 + g2 (GELU(LNmod2(x3) W1^T + b1) W2^T + b2)
        FF_TRY(gate(io.y2, base + 5 * H, p.dmods + base + 5 * H, G(pre + "mlp2.b")));
        FF_TRY(gemm1(gemm_wgrad(p.dy, H, io.u, F, H, F, Ri, G(pre + "mlp2.w"))));
        {
            GemmArgs g = gemm_dgrad(p.dy, H, W(pre + "mlp2.w"), Ri, F, H);
            g.epi.out0 = p.dbig; g.epi.ld0 = F;
            g.epi.gelu_pre = io.a1; g.epi.ld_pre = F;
            FF_TRY(gemm1(g));
        }
        FF_TRY(colsum(p.dbig, false, F, Ri, F, G(pre + "mlp1.b"), p.cs_ws, stream));
        FF_TRY(gemm1(gemm_wgrad(p.dbig, F, io.h2, H, F, H, Ri, G(pre + "mlp1.w"))));
        {
            GemmArgs g = gemm_dgrad(p.dbig, F, W(pre + "mlp1.w"), Ri, H, F);
            g.epi.out_f32 = 1; g.epi.out0 = p.dh; g.epi.ld0 = H;
            FF_TRY(gemm1(g));
        }
        FF_TRY(lnmod(io.x3, base + 3 * H));

        // cross-attention half: x3 = x_mid + CrossAttn(LN(x_mid) w + b, text) (no gate)
        FF_TRY(f32_to_bf16(p.gx, p.dy, static_cast<int64_t>(Ri) * H, stream));
        FF_TRY(colsum(p.gx, true, H, Ri, H, G(pre + "cross_proj.b"), p.cs_ws, stream));
        FF_TRY(gemm1(gemm_wgrad(p.dy, H, io.oc, H, H, H, Ri, G(pre + "cross_proj.w"))));
        {
            GemmArgs g = gemm_dgrad(p.dy, H, W(pre + "cross_proj.w"), Ri, H, H);
            g.epi.out0 = p.dob; g.epi.ld0 = H;
            FF_TRY(gemm1(g));
        }
        {
            // dq of the latent queries into dy (free again), dk | dv of the text into dkv
            AttnBwdSpec a{};
            a.q[0] = AttnBwdQuerySeg{nullptr, 0, 0, nullptr, 0, nullptr, 0, nullptr, 0};
            a.q[1] = AttnBwdQuerySeg{io.qc, H, Ni, io.oc, H, p.dob, H, p.dy, H, io.oc_lo, H};
            a.kv[0] = AttnBwdKvSeg{io.kv, 2 * H, Nt, p.dkv, p.dkv + H, 2 * H};
            a.kv[1] = AttnBwdKvSeg{nullptr, 0, 0, nullptr, nullptr, 0};
            a.q_col = 0; a.k_col = 0; a.v_col = H;
            a.B = B; a.heads = heads; a.head_dim = d;
            a.lse = io.lse_c;
            FF_TRY(attention_backward_general(a, p.attn_ws, p.attn_ws_bytes, stream));
        }
        {
            // RMSNorm backward of the cross q (latent rows) and of the text's k
            QkBwdArgs a{};
            a.rows_txt = 0; a.heads = heads; a.head_dim = d; a.sets = 1;
            a.rope_cs = nullptr; a.n_img = Ni; a.grid_f = c.grid_f; a.grid_h = c.grid_h; a.grid_w = c.grid_w;
            a.axes0 = c.rope_axes[0]; a.axes1 = c.rope_axes[1]; a.axes2 = c.rope_axes[2];
            a.part = p.part;
            int ct = 0, ci = 0;
            a.d = p.dy; a.ldd = H; a.raw = io.qc_raw; a.ldr = H; a.rows = Ri;
            a.q_scale_txt = a.q_scale_img = a.k_scale_txt = a.k_scale_img = W(pre + "cross_q_norm.scale");
            FF_TRY(qk_norm_rope_backward(a, &ct, &ci, stream));
            FF_TRY(reduce({total(ct + ci, 0, 2 * d, d, G(pre + "cross_q_norm.scale"))}));
            a.d = p.dkv; a.ldd = 2 * H; a.raw = io.kv_raw; a.ldr = 2 * H; a.rows = Rt;
            a.q_scale_txt = a.q_scale_img = a.k_scale_txt = a.k_scale_img = W(pre + "cross_k_norm.scale");
            FF_TRY(qk_norm_rope_backward(a, &ct, &ci, stream));
            FF_TRY(reduce({total(ct + ci, 0, 2 * d, d, G(pre + "cross_k_norm.scale"))}));
        }
        FF_TRY(colsum(p.dy, false, H, Ri, H, G(pre + "cross_q.b"), p.cs_ws, stream));
        FF_TRY(gemm1(gemm_wgrad(p.dy, H, io.hc, H, H, H, Ri, G(pre + "cross_q.w"))));
        {
            GemmArgs g = gemm_dgrad(p.dy, H, W(pre + "cross_q.w"), Ri, H, H);
            g.epi.out_f32 = 1; g.epi.out0 = p.dh; g.epi.ld0 = H;
            FF_TRY(gemm1(g));
        }
        FF_TRY(colsum(p.dkv, false, 2 * H, Rt, 2 * H, G(pre + "cross_kv.b"), p.cs_ws, stream));
        FF_TRY(gemm1(gemm_wgrad(p.dkv, 2 * H, f.txth, H, 2 * H, H, Rt, G(pre + "cross_kv.w"))));
        {
            // the embedded text's gradient: dtxt += d(k | v) W_kv
            GemmArgs g = gemm_dgrad(p.dkv, 2 * H, W(pre + "cross_kv.w"), Rt, H, 2 * H);
            g.epi.epi = EPI_GATED_RESIDUAL; g.epi.resid = p.dtxt; g.epi.ld_resid = H;
            g.epi.gate = nullptr; g.epi.rows_per_sample = Nt;
            FF_TRY(gemm1(g));
        }
        {
            const BwdSegs s = bwd_segs(&img, 1, B);
            FF_TRY(ln_modulate_backward(io.xmid, p.dh, p.gx, H, nullptr, 0, s, H, p.part, stream,
                                        W(pre + "cross_norm.scale")));
            FF_TRY(reduce({total(B * cps, 0, 2 * H, H, G(pre + "cross_norm.b")),
                           total(B * cps, H, 2 * H, H, G(pre + "cross_norm.scale"))}));
        }

        // self-attention half: x_mid = x_in + g1 (Attn(...) W_p^T + b_p)
        FF_TRY(gate(io.y1, base + 2 * H, p.dmods + base + 2 * H, G(pre + "proj.b")));
        FF_TRY(gemm1(gemm_wgrad(p.dy, H, io.o, H, H, H, Ri, G(pre + "proj.w"))));
        {
            GemmArgs g = gemm_dgrad(p.dy, H, W(pre + "proj.w"), Ri, H, H);
            g.epi.out0 = p.dob; g.epi.ld0 = H;
            FF_TRY(gemm1(g));
        }
        {
            const AttnBwdSeg s0{nullptr, 0, nullptr, nullptr, 0, nullptr, 0, 0, 0};
            const AttnBwdSeg s1{io.qkv, W3, io.o, p.dob, H, p.dbig, W3, Ni, H, io.o_lo, H};
            FF_TRY(attention_backward(s0, s1, B, heads, d, io.lse, p.attn_ws, p.attn_ws_bytes, stream));
        }
        {
            QkBwdArgs a{};
            a.d = p.dbig; a.ldd = W3; a.raw = io.raw; a.ldr = W3;
            a.rows_txt = 0; a.rows = Ri; a.heads = heads; a.head_dim = d;
            a.q_scale_txt = a.q_scale_img = W(pre + "q_norm.scale");
            a.k_scale_txt = a.k_scale_img = W(pre + "k_norm.scale");
            a.rope_cs = f.rope; a.n_img = Ni; a.grid_f = c.grid_f; a.grid_h = c.grid_h; a.grid_w = c.grid_w;
            a.axes0 = c.rope_axes[0]; a.axes1 = c.rope_axes[1]; a.axes2 = c.rope_axes[2];
            a.part = p.part;
            int ct = 0, ci = 0;
            FF_TRY(qk_norm_rope_backward(a, &ct, &ci, stream));
            FF_TRY(reduce({total(ct + ci, 0, 2 * d, d, G(pre + "q_norm.scale")),
                           total(ct + ci, d, 2 * d, d, G(pre + "k_norm.scale"))}));
        }
        FF_TRY(colsum(p.dbig, false, W3, Ri, W3, G(pre + "qkv.b"), p.cs_ws, stream));
        FF_TRY(gemm1(gemm_wgrad(p.dbig, W3, io.h1, H, W3, H, Ri, G(pre + "qkv.w"))));
        {
            GemmArgs g = gemm_dgrad(p.dbig, W3, W(pre + "qkv.w"), Ri, H, W3);
            g.epi.out_f32 = 1; g.epi.out0 = p.dh; g.epi.ld0 = H;
            FF_TRY(gemm1(g));
        }
        FF_TRY(lnmod(io.xin, base));
    }

    // ---- patch embedding (gx now holds dL/dx after it)
    FF_TRY(f32_to_bf16(p.gx, p.dy, static_cast<int64_t>(Ri) * H, stream));
    FF_TRY(gemm1(gemm_wgrad(p.dy, H, f.xb, P, H, P, Ri, G("img_in.w"))));
    FF_TRY(colsum(p.gx, true, H, Ri, H, G("img_in.b"), p.cs_ws, stream));
    if (dx_t) {
        GemmArgs g = gemm_dgrad(p.dy, H, W("img_in.w"), Ri, P, H);
        g.epi.out_f32 = 1; g.epi.out0 = dx_t; g.epi.ld0 = P;
        FF_TRY(gemm1(g));
    }

    // ---- text MLP: txth = GELU(txt W_1^T + b_1) W_2^T + b_2
    FF_TRY(f32_to_bf16(p.dtxt, p.dyt, static_cast<int64_t>(Rt) * H, stream));
    FF_TRY(colsum(p.dtxt, true, H, Rt, H, G("txt_in2.b"), p.cs_ws, stream));
    FF_TRY(gemm1(gemm_wgrad(p.dyt, H, f.txt1, H, H, H, Rt, G("txt_in2.w"))));
    {
        GemmArgs g = gemm_dgrad(p.dyt, H, W("txt_in2.w"), Rt, H, H);
        g.epi.out0 = p.dkv; g.epi.ld0 = H;
        g.epi.gelu_pre = f.txt_pre; g.epi.ld_pre = H;
        FF_TRY(gemm1(g));
    }
    FF_TRY(colsum(p.dkv, false, H, Rt, H, G("txt_in.b"), p.cs_ws, stream));
    FF_TRY(gemm1(gemm_wgrad(p.dkv, H, txt, c.txt_dim, H, c.txt_dim, Rt, G("txt_in.w"))));

    // ---- shared modulation, SiLU(e), the timestep MLP (B rows, padded to Kp for the products)
    {
        const int64_t stride = L > 1 ? model_offset(m, "blocks.1.mod.b") - model_offset(m, "blocks.0.mod.b") : 0;
        FF_TRY(wan_modulation_backward(p.dmods, Wm, B, Kp, H, L, G("blocks.0.mod.b"), stride, G("final.mod.b"), p.de0,
                                       p.de0_b, p.de_fin, stream));
    }
    // Linears of B rows: HBM-bound kernels up to kRowsMaxB rows, the
    // tensor-core GEMM over Kp padded rows beyond
    const bool few = B <= kRowsMaxB;
    if (few) FF_TRY(rows_wgrad(B, 6 * H, H, p.de0, 6 * H, f.tc, H, G("mod.w"), H, stream));
    else FF_TRY(gemm1(gemm_wgrad(p.de0_b, 6 * H, f.tc, H, 6 * H, H, Kp, G("mod.w"))));
    FF_TRY(colsum(p.de0, true, 6 * H, B, 6 * H, G("mod.b"), p.cs_ws, stream));
    if (few) {
        FF_TRY(rows_dgrad(B, 6 * H, H, p.de0, 6 * H, W("mod.w"), H, p.dtc, H, p.rows_part, p.rows_part_floats,
                          stream));
    } else {
        GemmArgs g = gemm_dgrad(p.de0_b, 6 * H, W("mod.w"), Kp, H, 6 * H);
        g.epi.out_f32 = 1; g.epi.out0 = p.dtc; g.epi.ld0 = H;
        FF_TRY(gemm1(g));
    }
    // d e = d SiLU(e) SiLU'(e) + the final layer's shift and scale gradients
    FF_TRY(silu_backward(p.dtc, H, f.pre_c, B, Kp, H, p.dc, p.dc_b, stream, p.de_fin));
    if (few) FF_TRY(rows_wgrad(B, H, H, p.dc, H, f.th, H, G("t_embed.fc2.w"), H, stream));
    else FF_TRY(gemm1(gemm_wgrad(p.dc_b, H, f.th, H, H, H, Kp, G("t_embed.fc2.w"))));
    FF_TRY(colsum(p.dc, true, H, B, H, G("t_embed.fc2.b"), p.cs_ws, stream));
    if (few) {
        FF_TRY(rows_dgrad(B, H, H, p.dc, H, W("t_embed.fc2.w"), H, p.dth, H, p.rows_part, p.rows_part_floats,
                          stream));
    } else {
        GemmArgs g = gemm_dgrad(p.dc_b, H, W("t_embed.fc2.w"), Kp, H, H);
        g.epi.out_f32 = 1; g.epi.out0 = p.dth; g.epi.ld0 = H;
        FF_TRY(gemm1(g));
    }
    FF_TRY(silu_backward(p.dth, H, f.pre_fc1, B, Kp, H, p.da, p.da_b, stream));
    if (few) FF_TRY(rows_wgrad(B, H, tf, p.da, H, f.temb, tf, G("t_embed.fc1.w"), tf, stream));
    else FF_TRY(gemm1(gemm_wgrad(p.da_b, H, f.temb, tf, H, tf, Kp, G("t_embed.fc1.w"))));
    return colsum(p.da, true, H, B, H, G("t_embed.fc1.b"), p.cs_ws, stream);
}

}  // namespace ff
