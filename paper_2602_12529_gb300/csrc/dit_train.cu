// dit_train.cu -- the training pass of the MMDiT velocity (the forward that
// every GRPO-style trainer runs "again for training", and its gradient):
//   ff_dit_forward_train  the velocity call of ff_dit_velocity over one
//                         buffer set per block, keeping every value the
//                         backward reads (bit-identical v);
//   ff_dit_backward       from dL/dv to dL/dtheta for every weight (an fp32
//                         blob laid out like the weight blob) and dL/dx_t.
//
// The backward runs the blocks in reverse.  Per Linear y = x W^T + b it
// issues the weight-gradient product dW = dy^T x (both operands MN-major,
// K = tokens) and the input-gradient product dx = dy W (W as an MN-major B
// operand) on the tcgen05 GEMM, with the GELU derivative fused into the
// MLP's input-gradient epilogue; the gated residuals, LN-modulations and the
// QK-RMSNorm + RoPE go backward in backward.cu's row kernels, and every sum
// over tokens (bias, gate, shift, scale and norm-scale gradients) is a
// fixed-order reduction of per-chunk partials, so the gradient is
// deterministic.
//
// Workspace (one caller buffer, written by the forward, read by the
// backward; R = B (N_t + N_i) rows, "stream-major" as in dit.cu):
//   mods fp32 [B, W_mod]; time-MLP operands temb / SiLU(fc1) / SiLU(c) bf16,
//   zero-padded to a multiple of 8 rows, and their pre-activation copies;
//   per double-stream block: x_in, x_mid fp32 [R, H]; h1, h2, o, y1, y2 bf16
//   [R, H]; raw and normalised qkv bf16 [R, 3H]; a1 = MLP1 + bias and
//   u = GELU(a1) bf16 [R, F]; the attention log-sum-exp and the bf16
//   rounding residual of its output (bf16 [R, H]: the backward's
//   D = rowsum(dO O) is formed from O to about 16 bits);
//   per single-stream block: x_in fp32; h, y2 bf16 [R, H]; raw linear1 bf16
//   [R, 3H + F]; qkv bf16 [R, 3H]; u = [o | GELU(mlp)] bf16 [R, H + F]; o's
//   residual; lse;
//   the final residual and LN-modulate output; then the backward's scratch.
// In recompute mode (ff_dit_set_train_recompute) the blocks of each kind
// share one set of those activations and only the block inputs are kept,
// with (mode 1) each double block's joint-attention output, its low part and
// lse; the backward re-runs each block's forward (bit-identical: every kernel
// is deterministic) just before its backward, a double block's without its
// attention in mode 1.
#include <initializer_list>
#include <string>
#include <vector>

#include "internal.h"
#include "reduce_jobs.h"

namespace ff {
namespace {

constexpr size_t kAlign = 256;
size_t up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

struct TrainPlan {
    FwdBufs f;
    std::vector<DitBlockIo> blk;
    int rows_pad;
    // backward scratch
    float *gx, *dh, *part, *cs_ws;
    __nv_bfloat16 *dy, *dbig, *dqkv, *dob, *dvb;
    void* attn_ws;
    size_t attn_ws_bytes;
    float *dmods, *dtc, *dth, *dc, *da;
    float* rows_part;          // rows_dgrad's partial sums
    size_t rows_part_floats;
    __nv_bfloat16 *dmods_b, *dc_b, *da_b;
    size_t bytes;
};

TrainPlan plan(const ff_dit_config& c, int64_t Wm, int B, uint8_t* base, int recompute) {
    const size_t H = c.hidden, F = c.mlp, P = c.patch_dim, tf = c.time_freq_dim, d = c.head_dim;
    const size_t Nt = c.n_txt, Ni = static_cast<size_t>(c.grid_f) * c.grid_h * c.grid_w;
    const size_t Rt = B * Nt, Ri = B * Ni, R = Rt + Ri;
    const size_t Kp = (B + 7) / 8 * 8;
    size_t o = 0;
    auto take = [&](size_t bytes) { uint8_t* p = base ? base + o : nullptr; o += up(bytes); return p; };
    auto f32 = [&](size_t n) { return reinterpret_cast<float*>(take(n * 4)); };
    auto b16 = [&](size_t n) { return reinterpret_cast<__nv_bfloat16*>(take(n * 2)); };
    TrainPlan p{};
    p.rows_pad = static_cast<int>(Kp);
    FwdBufs& f = p.f;
    f.mods = f32(B * Wm);
    f.temb = b16(Kp * tf);
    f.th = b16(Kp * H);
    f.tc = b16(Kp * H);
    f.pre_fc1 = b16(B * H);
    f.pre_c = b16(B * H);
    f.xb = b16(Ri * P);
    f.rope = reinterpret_cast<float2*>(take(static_cast<size_t>(rope_table_size(
        c.grid_f, c.grid_h, c.grid_w, c.rope_axes[0], c.rope_axes[1], c.rope_axes[2])) * sizeof(float2)));
    f.attn_ws_bytes = attention_split_ws_bytes(c.head_dim);
    f.attn_ws = take(f.attn_ws_bytes);
    const int L = c.n_double + c.n_single;
    const size_t lse_n = static_cast<size_t>(B) * c.heads * attn_lse_rows(static_cast<int>(Nt), static_cast<int>(Ni));
    p.blk.resize(L);
    float* x = f32(R * H);
    f.x0 = x;
    // recompute: one activation set per block kind, shared by the blocks of
    // that kind (re-filled by the backward); kept per block: the input and,
    // in mode 1, a double block's joint-attention O, its low part and lse
    DitBlockIo shared_dbl{}, shared_sgl{};
    bool have_dbl = false, have_sgl = false;
    for (int l = 0; l < L; ++l) {
        DitBlockIo& io = p.blk[l];
        const bool dbl = l < c.n_double;
        if (recompute && (dbl ? have_dbl : have_sgl)) {
            io = dbl ? shared_dbl : shared_sgl;
            io.xin = x;
            if (!dbl) io.xmid = x;
            if (dbl && recompute == 1) {
                io.o = b16(R * H);
                io.o_lo = b16(R * H);
                io.lse = f32(lse_n);
            }
            x = f32(R * H);
            io.xout = x;
            continue;
        }
        io = DitBlockIo{};
        io.xin = x;
        io.h1 = b16(R * H);
        io.raw = b16(R * (dbl ? 3 * H : 3 * H + F));
        io.qkv = b16(R * 3 * H);
        io.lse = f32(lse_n);
        io.o_lo = b16(R * H);
        if (dbl) {
            io.o = b16(R * H);
            io.y1 = b16(R * H);
            io.xmid = f32(R * H);
            io.h2 = b16(R * H);
            io.a1 = b16(R * F);
            io.u = b16(R * F);
        } else {
            io.xmid = io.xin;
            io.u = b16(R * (H + F));
        }
        io.y2 = b16(R * H);
        x = f32(R * H);
        io.xout = x;
        if (dbl) { shared_dbl = io; have_dbl = true; }
        else { shared_sgl = io; have_sgl = true; }
    }
    f.xfin = x;
    f.hf = b16(Ri * H);
    f.blocks = nullptr;   // set by the caller once the plan has its final address

    const size_t wide = c.n_single ? 3 * H + F : F;
    p.gx = f32(R * H);
    p.dh = f32(R * H);
    p.dy = b16(R * H);
    p.dbig = b16(R * wide);
    p.dqkv = b16(R * 3 * H);
    p.dob = b16(R * H);
    p.dvb = b16(Ri * P);
    const size_t chunks = static_cast<size_t>(B) * (bwd_chunks(static_cast<int>(Nt)) + bwd_chunks(static_cast<int>(Ni)));
    const size_t qk_ctas = (Rt + kQkBwdRows - 1) / kQkBwdRows + (Ri + kQkBwdRows - 1) / kQkBwdRows;
    p.part = f32(std::max(chunks * 2 * H, qk_ctas * 2 * d));
    size_t cs = colsum_ws_floats(static_cast<int>(R), static_cast<int>(std::max(wide, 3 * H)));
    cs = std::max(cs, colsum_ws_floats(B, static_cast<int>(Wm)));
    cs = std::max(cs, colsum_ws_floats(static_cast<int>(Ri), static_cast<int>(std::max(H, P))));
    p.cs_ws = f32(cs);
    p.attn_ws_bytes = attention_backward_ws_bytes(B, c.heads, static_cast<int>(Nt), static_cast<int>(Ni));
    p.attn_ws = take(p.attn_ws_bytes);
    p.dmods = f32(B * Wm);
    p.dmods_b = b16(Kp * Wm);
    p.dtc = f32(Kp * H);
    p.dth = f32(Kp * H);
    p.dc = f32(B * H);
    p.da = f32(B * H);
    p.dc_b = b16(Kp * H);
    p.da_b = b16(Kp * H);
    p.rows_part_floats = B <= kRowsMaxB ? static_cast<size_t>(rows_dgrad_chunks(static_cast<int>(Wm))) * B * H : 0;
    p.rows_part = f32(p.rows_part_floats);
    p.bytes = o;
    return p;
}

int check_model(const ff_dit* m, int B) {
    if (!m) return set_error(FF_ERR_INVALID_ARG, "model is null");
    if (B <= 0) return set_error(FF_ERR_INVALID_ARG, "B=%d must be positive", B);
    const ff_dit_config& c = model_config(m);

    const int64_t Ni = static_cast<int64_t>(c.grid_f) * c.grid_h * c.grid_w;
    if ((static_cast<int64_t>(B) * c.n_txt) % 8 || (B * Ni) % 8)
        return set_error(FF_ERR_UNSUPPORTED, "training pass: B N_t and B N_i must be multiples of 8");
    return FF_OK;
}

GemmArgs wgrad(const void* dy, int64_t lddy, const void* x, int64_t ldx, int M, int N, int K, float* out) {
    return gemm_wgrad(dy, lddy, x, ldx, M, N, K, out);
}
GemmArgs dgrad(const void* dy, int64_t lddy, const void* w, int M, int N, int K) {
    return gemm_dgrad(dy, lddy, w, M, N, K);
}

}  // namespace
}  // namespace ff

extern "C" {

int ff_dit_train_workspace_size(const ff_dit* m, int B, size_t* bytes) {
    using namespace ff;
    FF_TRY(check_model(m, B));
    if (!bytes) return set_error(FF_ERR_INVALID_ARG, "bytes is null");
    *bytes = model_config(m).arch == FF_ARCH_WAN
                 ? wan_train_workspace_bytes(m, B)
                 : plan(model_config(m), model_mod_width(m), B, nullptr, model_train_recompute(m)).bytes;
    return FF_OK;
}

int ff_dit_forward_train(const ff_dit* m, int B, const float* x_t, const void* txt, const float* t, float* v_out,
                         void* ws, size_t ws_bytes, cudaStream_t stream) {
    using namespace ff;
    FF_TRY(check_model(m, B));
    if (!x_t || !txt || !t || !v_out || !ws) return set_error(FF_ERR_INVALID_ARG, "null pointer argument");
    if (!aligned16(x_t) || !aligned16(txt) || !aligned16(v_out) || (reinterpret_cast<uintptr_t>(ws) % kAlign))
        return set_error(FF_ERR_INVALID_ARG, "misaligned pointer (arrays 16 B, workspace 256 B)");
    const ff_dit_config& c = model_config(m);
    model_note_forward_train(m);
    if (c.arch == FF_ARCH_WAN) return wan_forward_train(m, B, x_t, txt, t, v_out, ws, ws_bytes, stream);
    TrainPlan p = plan(c, model_mod_width(m), B, static_cast<uint8_t*>(ws), model_train_recompute(m));
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
    return mmdit_forward(m, B, x_t, txt, t, v_out, p.f, stream);
}

int ff_dit_backward(const ff_dit* m, int B, const void* txt, const float* dv, float* grad, float* dx_t, void* ws,
                    size_t ws_bytes, cudaStream_t stream) {
    using namespace ff;
    FF_TRY(check_model(m, B));
    if (!txt || !dv || !grad || !ws) return set_error(FF_ERR_INVALID_ARG, "null pointer argument");
    if (!aligned16(txt) || !aligned16(dv) || !aligned16(grad) || (dx_t && !aligned16(dx_t)) ||
        (reinterpret_cast<uintptr_t>(ws) % kAlign))
        return set_error(FF_ERR_INVALID_ARG, "misaligned pointer (arrays 16 B, workspace 256 B)");
    const ff_dit_config& c = model_config(m);
    if (model_forward_train_mode(m) != model_train_recompute(m))
        return set_error(FF_ERR_INVALID_ARG, model_forward_train_mode(m) < 0
                                                 ? "backward: no ff_dit_forward_train on this model yet"
                                                 : "backward: recompute mode changed since ff_dit_forward_train");
    if (c.arch == FF_ARCH_WAN) return wan_backward(m, B, txt, dv, grad, dx_t, ws, ws_bytes, stream);
    const int64_t Wm = model_mod_width(m);
    const int recompute = model_train_recompute(m);
    TrainPlan p = plan(c, Wm, B, static_cast<uint8_t*>(ws), recompute);
    if (!model_attention_split(m)) p.f.attn_ws = nullptr;
    if (ws_bytes < p.bytes) return set_error(FF_ERR_WORKSPACE, "workspace %zu B < %zu B needed", ws_bytes, p.bytes);
    const FwdBufs& f = p.f;
    const int H = c.hidden, F = c.mlp, P = c.patch_dim, d = c.head_dim, heads = c.heads, tf = c.time_freq_dim;
    const int Nt = c.n_txt, Ni = c.grid_f * c.grid_h * c.grid_w;
    const int Rt = B * Nt, Ri = B * Ni, R = Rt + Ri;
    const int Kp = p.rows_pad;
    const int cps_t = bwd_chunks(Nt), cps_i = bwd_chunks(Ni);
    const __nv_bfloat16* w0 = model_weights(m);
    auto W = [&](const std::string& n) { return w0 + model_offset(m, n.c_str()); };
    auto G = [&](const std::string& n) { return grad + model_offset(m, n.c_str()); };
    auto group = [&](GemmArgs* g, int n) { return gemm_bf16_group(g, n, stream); };
    // reductions of chunk partials (columns ncols of part at offset col),
    // the ones that follow one backward kernel batched into one launch
    auto per_sample = [&](int first, int count, int col, float* out) {
        return ReduceJob{p.part + col, 2 * H, H, chunk_span(first, count), 1, out, Wm};
    };
    auto total = [&](int first, int count, int col, int64_t ld, int ncols, float* out) {
        return ReduceJob{p.part + col, ld, ncols, chunk_span(first, count), 0, out, 0};
    };
    auto reduce = [&](std::initializer_list<ReduceJob> jobs) {
        return reduce_chunks_batch(jobs.begin(), static_cast<int>(jobs.size()), B, stream);
    };

    // ---- final layer: v = LNmod(x_img) W_f^T + b_f
    const int64_t off_f = static_cast<int64_t>(c.n_double) * 12 * H + static_cast<int64_t>(c.n_single) * 3 * H;
    FF_TRY(f32_to_bf16(dv, p.dvb, static_cast<int64_t>(Ri) * P, stream));
    {
        GemmArgs g = wgrad(p.dvb, P, f.hf, H, P, H, Ri, G("final.w"));
        FF_TRY(group(&g, 1));
    }
    FF_TRY(colsum(dv, true, P, Ri, P, G("final.b"), p.cs_ws, stream));
    {
        GemmArgs g = dgrad(p.dvb, P, W("final.w"), Ri, H, P);
        g.epi.out_f32 = 1; g.epi.out0 = p.dh + static_cast<int64_t>(Rt) * H; g.epi.ld0 = H;
        FF_TRY(group(&g, 1));
    }
    if (cudaMemsetAsync(p.gx, 0, static_cast<size_t>(R) * H * 4, stream) != cudaSuccess)
        return set_error(FF_ERR_CUDA, "backward: memset failed");
    {
        const BwdSeg sg{Rt, Ni, 0, static_cast<int>(off_f + H)};
        const BwdSegs s = bwd_segs(&sg, 1, B);
        FF_TRY(ln_modulate_backward(f.xfin, p.dh, p.gx, H, f.mods, Wm, s, H, p.part, stream));
        FF_TRY(reduce({per_sample(0, cps_i, 0, p.dmods + off_f), per_sample(0, cps_i, H, p.dmods + off_f + H)}));
    }

    // ---- single-stream blocks, last first
    for (int l = c.n_single - 1; l >= 0; --l) {
        const DitBlockIo& io = p.blk[c.n_double + l];
        if (recompute) FF_TRY(mmdit_forward_single(m, B, l, io, f, stream));
        const int off = static_cast<int>(static_cast<int64_t>(c.n_double) * 12 * H + static_cast<int64_t>(l) * 3 * H);
        const std::string pre = "single." + std::to_string(l) + ".";
        const int W1 = 3 * H + F;
        // gated residual: dy = g gate, gate and linear2 bias gradients
        {
            const BwdSeg sg[2] = {{0, Nt, off + 2 * H, 0}, {Rt, Ni, off + 2 * H, 0}};
            const BwdSegs s = bwd_segs(sg, 2, B);
            FF_TRY(gate_backward(p.gx, io.y2, H, f.mods, Wm, s, H, p.dy, p.part, stream));
            ChunkSpans sp{};
            sp.n = 2; sp.first[0] = 0; sp.count[0] = cps_t; sp.first[1] = s.first[1]; sp.count[1] = cps_i;
            ChunkSpans all = sp;
            all.count[0] = B * cps_t; all.count[1] = B * cps_i;
            FF_TRY(reduce({ReduceJob{p.part, 2 * H, H, sp, 1, p.dmods + off + 2 * H, Wm},
                           ReduceJob{p.part + H, 2 * H, H, all, 0, G(pre + "linear2.b"), 0}}));
        }
        {
            GemmArgs g = wgrad(p.dy, H, io.u, H + F, H, H + F, R, G(pre + "linear2.w"));
            FF_TRY(group(&g, 1));
        }
        {
            // d[o | GELU(m)] = dy W2: the attention part to dob, the MLP part
            // (times GELU'(m)) straight into the linear1 gradient's columns 3H..
            GemmArgs g = dgrad(p.dy, H, W(pre + "linear2.w"), R, H + F, H);
            GemmEpilogue& e = g.epi;
            e.out0 = p.dob; e.ld0 = H;
            e.split_n = H; e.out1 = p.dbig; e.ld1 = W1; e.col1 = 3 * H;
            e.gelu_pre = io.raw + 3 * H; e.ld_pre = W1; e.act_from = H;
            FF_TRY(group(&g, 1));
        }
        {
            AttnBwdSeg s0{io.qkv, 3 * H, io.u, p.dob, H + F, p.dbig, W1, Nt, H, io.o_lo, H};
            AttnBwdSeg s1{io.qkv + static_cast<int64_t>(Rt) * 3 * H, 3 * H, io.u + static_cast<int64_t>(Rt) * (H + F),
                          p.dob + static_cast<int64_t>(Rt) * H, H + F, p.dbig + static_cast<int64_t>(Rt) * W1, W1, Ni, H,
                          io.o_lo + static_cast<int64_t>(Rt) * H, H};
            FF_TRY(attention_backward(s0, s1, B, heads, d, io.lse, p.attn_ws, p.attn_ws_bytes, stream));
        }
        {
            QkBwdArgs a{};
            a.d = p.dbig; a.ldd = W1; a.raw = io.raw; a.ldr = W1;
            a.rows_txt = Rt; a.rows = R; a.heads = heads; a.head_dim = d;
            a.q_scale_txt = a.q_scale_img = W(pre + "q_norm.scale");
            a.k_scale_txt = a.k_scale_img = W(pre + "k_norm.scale");
            a.rope_cs = f.rope; a.n_img = Ni; a.grid_f = c.grid_f; a.grid_h = c.grid_h; a.grid_w = c.grid_w;
            a.axes0 = c.rope_axes[0]; a.axes1 = c.rope_axes[1]; a.axes2 = c.rope_axes[2];
            a.part = p.part;
            int ct = 0, ci = 0;
            FF_TRY(qk_norm_rope_backward(a, &ct, &ci, stream));
            FF_TRY(reduce({total(0, ct + ci, 0, 2 * d, d, G(pre + "q_norm.scale")),
                           total(0, ct + ci, d, 2 * d, d, G(pre + "k_norm.scale"))}));
        }
        FF_TRY(colsum(p.dbig, false, W1, R, W1, G(pre + "linear1.b"), p.cs_ws, stream));
        {
            GemmArgs g = wgrad(p.dbig, W1, io.h1, H, W1, H, R, G(pre + "linear1.w"));
            FF_TRY(group(&g, 1));
        }
        {
            GemmArgs g = dgrad(p.dbig, W1, W(pre + "linear1.w"), R, H, W1);
            g.epi.out_f32 = 1; g.epi.out0 = p.dh; g.epi.ld0 = H;
            FF_TRY(group(&g, 1));
        }
        {
            const BwdSeg sg[2] = {{0, Nt, 0, off + H}, {Rt, Ni, 0, off + H}};
            const BwdSegs s = bwd_segs(sg, 2, B);
            FF_TRY(ln_modulate_backward(io.xin, p.dh, p.gx, H, f.mods, Wm, s, H, p.part, stream));
            ChunkSpans sp{};
            sp.n = 2; sp.first[0] = 0; sp.count[0] = cps_t; sp.first[1] = s.first[1]; sp.count[1] = cps_i;
            FF_TRY(reduce({ReduceJob{p.part, 2 * H, H, sp, 1, p.dmods + off, Wm},
                           ReduceJob{p.part + H, 2 * H, H, sp, 1, p.dmods + off + H, Wm}}));
        }
    }

    // ---- double-stream blocks, last first (image problem first in each grouped launch)
    struct Stream { const char* name; int row0, rows, tokens, mod, first, cps; };
    for (int l = c.n_double - 1; l >= 0; --l) {
        const DitBlockIo& io = p.blk[l];
        if (recompute) {
            DitBlockIo r = io;
            r.attn_kept = recompute == 1;   // mode 1: the joint attention's outputs were kept
            FF_TRY(mmdit_forward_double(m, B, l, r, f, stream));
        }
        const int base = l * 12 * H;
        const int first_img = B * cps_t;
        const Stream st[2] = {{"img", Rt, Ri, Ni, base, first_img, cps_i}, {"txt", 0, Rt, Nt, base + 6 * H, 0, cps_t}};
        const std::string pre = "double." + std::to_string(l) + ".";
        auto P_ = [&](const Stream& s, const char* n) { return pre + s.name + "." + n; };
        const BwdSeg seg_txt{0, Nt, 0, 0}, seg_img{Rt, Ni, 0, 0};
        // gate backward of a gated branch (y = pre-gate values, gate at mod + k H)
        auto gate = [&](const __nv_bfloat16* y, int k, const char* bias) {
            BwdSeg sg[2] = {seg_txt, seg_img};
            sg[0].col_a = st[1].mod + k * H;
            sg[1].col_a = st[0].mod + k * H;
            const BwdSegs s = bwd_segs(sg, 2, B);
            FF_TRY(gate_backward(p.gx, y, H, f.mods, Wm, s, H, p.dy, p.part, stream));
            return reduce({per_sample(st[0].first, st[0].cps, 0, p.dmods + st[0].mod + k * H),
                           total(st[0].first, B * st[0].cps, H, 2 * H, H, G(P_(st[0], bias))),
                           per_sample(st[1].first, st[1].cps, 0, p.dmods + st[1].mod + k * H),
                           total(st[1].first, B * st[1].cps, H, 2 * H, H, G(P_(st[1], bias)))});
        };
        auto lnmod = [&](const float* x, int k_shift) {
            BwdSeg sg[2] = {seg_txt, seg_img};
            sg[0].col_b = st[1].mod + (k_shift + 1) * H;
            sg[1].col_b = st[0].mod + (k_shift + 1) * H;
            const BwdSegs s = bwd_segs(sg, 2, B);
            FF_TRY(ln_modulate_backward(x, p.dh, p.gx, H, f.mods, Wm, s, H, p.part, stream));
            return reduce({per_sample(st[0].first, st[0].cps, 0, p.dmods + st[0].mod + k_shift * H),
                           per_sample(st[0].first, st[0].cps, H, p.dmods + st[0].mod + (k_shift + 1) * H),
                           per_sample(st[1].first, st[1].cps, 0, p.dmods + st[1].mod + k_shift * H),
                           per_sample(st[1].first, st[1].cps, H, p.dmods + st[1].mod + (k_shift + 1) * H)});
        };
        // MLP half: x_out = x_mid + gate2 (GELU(LNmod2(x_mid) W1^T + b1) W2^T + b2)
        FF_TRY(gate(io.y2, 5, "mlp2.b"));
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i)
                g[i] = wgrad(p.dy + static_cast<int64_t>(st[i].row0) * H, H, io.u + static_cast<int64_t>(st[i].row0) * F,
                             F, H, F, st[i].rows, G(P_(st[i], "mlp2.w")));
            FF_TRY(group(g, 2));
        }
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i) {
                g[i] = dgrad(p.dy + static_cast<int64_t>(st[i].row0) * H, H, W(P_(st[i], "mlp2.w")), st[i].rows, F, H);
                g[i].epi.out0 = p.dbig + static_cast<int64_t>(st[i].row0) * F; g[i].epi.ld0 = F;
                g[i].epi.gelu_pre = io.a1 + static_cast<int64_t>(st[i].row0) * F; g[i].epi.ld_pre = F;
            }
            FF_TRY(group(g, 2));
        }
        for (const Stream& s : st)
            FF_TRY(colsum(p.dbig + static_cast<int64_t>(s.row0) * F, false, F, s.rows, F, G(P_(s, "mlp1.b")), p.cs_ws,
                          stream));
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i)
                g[i] = wgrad(p.dbig + static_cast<int64_t>(st[i].row0) * F, F, io.h2 + static_cast<int64_t>(st[i].row0) * H,
                             H, F, H, st[i].rows, G(P_(st[i], "mlp1.w")));
            FF_TRY(group(g, 2));
        }
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i) {
                g[i] = dgrad(p.dbig + static_cast<int64_t>(st[i].row0) * F, F, W(P_(st[i], "mlp1.w")), st[i].rows, H, F);
                g[i].epi.out_f32 = 1; g[i].epi.out0 = p.dh + static_cast<int64_t>(st[i].row0) * H; g[i].epi.ld0 = H;
            }
            FF_TRY(group(g, 2));
        }
        FF_TRY(lnmod(io.xmid, 3));
        // attention half: x_mid = x_in + gate1 (attn(...) W_p^T + b_p)
        FF_TRY(gate(io.y1, 2, "proj.b"));
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i)
                g[i] = wgrad(p.dy + static_cast<int64_t>(st[i].row0) * H, H, io.o + static_cast<int64_t>(st[i].row0) * H,
                             H, H, H, st[i].rows, G(P_(st[i], "proj.w")));
            FF_TRY(group(g, 2));
        }
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i) {
                g[i] = dgrad(p.dy + static_cast<int64_t>(st[i].row0) * H, H, W(P_(st[i], "proj.w")), st[i].rows, H, H);
                g[i].epi.out0 = p.dob + static_cast<int64_t>(st[i].row0) * H; g[i].epi.ld0 = H;
            }
            FF_TRY(group(g, 2));
        }
        {
            AttnBwdSeg s0{io.qkv, 3 * H, io.o, p.dob, H, p.dqkv, 3 * H, Nt, 0, io.o_lo, H};
            AttnBwdSeg s1{io.qkv + static_cast<int64_t>(Rt) * 3 * H, 3 * H, io.o + static_cast<int64_t>(Rt) * H,
                          p.dob + static_cast<int64_t>(Rt) * H, H, p.dqkv + static_cast<int64_t>(Rt) * 3 * H, 3 * H, Ni, 0,
                          io.o_lo + static_cast<int64_t>(Rt) * H, H};
            FF_TRY(attention_backward(s0, s1, B, heads, d, io.lse, p.attn_ws, p.attn_ws_bytes, stream));
        }
        {
            QkBwdArgs a{};
            a.d = p.dqkv; a.ldd = 3 * H; a.raw = io.raw; a.ldr = 3 * H;
            a.rows_txt = Rt; a.rows = R; a.heads = heads; a.head_dim = d;
            a.q_scale_txt = W(pre + "txt.q_norm.scale"); a.k_scale_txt = W(pre + "txt.k_norm.scale");
            a.q_scale_img = W(pre + "img.q_norm.scale"); a.k_scale_img = W(pre + "img.k_norm.scale");
            a.rope_cs = f.rope; a.n_img = Ni; a.grid_f = c.grid_f; a.grid_h = c.grid_h; a.grid_w = c.grid_w;
            a.axes0 = c.rope_axes[0]; a.axes1 = c.rope_axes[1]; a.axes2 = c.rope_axes[2];
            a.part = p.part;
            int ct = 0, ci = 0;
            FF_TRY(qk_norm_rope_backward(a, &ct, &ci, stream));
            FF_TRY(reduce({total(0, ct, 0, 2 * d, d, G(pre + "txt.q_norm.scale")),
                           total(0, ct, d, 2 * d, d, G(pre + "txt.k_norm.scale")),
                           total(ct, ci, 0, 2 * d, d, G(pre + "img.q_norm.scale")),
                           total(ct, ci, d, 2 * d, d, G(pre + "img.k_norm.scale"))}));
        }
        for (const Stream& s : st)
            FF_TRY(colsum(p.dqkv + static_cast<int64_t>(s.row0) * 3 * H, false, 3 * H, s.rows, 3 * H, G(P_(s, "qkv.b")),
                          p.cs_ws, stream));
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i)
                g[i] = wgrad(p.dqkv + static_cast<int64_t>(st[i].row0) * 3 * H, 3 * H,
                             io.h1 + static_cast<int64_t>(st[i].row0) * H, H, 3 * H, H, st[i].rows, G(P_(st[i], "qkv.w")));
            FF_TRY(group(g, 2));
        }
        {
            GemmArgs g[2];
            for (int i = 0; i < 2; ++i) {
                g[i] = dgrad(p.dqkv + static_cast<int64_t>(st[i].row0) * 3 * H, 3 * H, W(P_(st[i], "qkv.w")), st[i].rows,
                             H, 3 * H);
                g[i].epi.out_f32 = 1; g[i].epi.out0 = p.dh + static_cast<int64_t>(st[i].row0) * H; g[i].epi.ld0 = H;
            }
            FF_TRY(group(g, 2));
        }
        FF_TRY(lnmod(io.xin, 0));
    }

    // ---- embeddings (gx now holds dL/dx after the embeddings)
    FF_TRY(f32_to_bf16(p.gx, p.dy, static_cast<int64_t>(R) * H, stream));
    {
        GemmArgs g = wgrad(p.dy + static_cast<int64_t>(Rt) * H, H, f.xb, P, H, P, Ri, G("img_in.w"));
        FF_TRY(group(&g, 1));
    }
    FF_TRY(colsum(p.gx + static_cast<int64_t>(Rt) * H, true, H, Ri, H, G("img_in.b"), p.cs_ws, stream));
    {
        GemmArgs g = wgrad(p.dy, H, txt, c.txt_dim, H, c.txt_dim, Rt, G("txt_in.w"));
        FF_TRY(group(&g, 1));
    }
    FF_TRY(colsum(p.gx, true, H, Rt, H, G("txt_in.b"), p.cs_ws, stream));
    if (dx_t) {
        GemmArgs g = dgrad(p.dy + static_cast<int64_t>(Rt) * H, H, W("img_in.w"), Ri, P, H);
        g.epi.out_f32 = 1; g.epi.out0 = dx_t; g.epi.ld0 = P;
        FF_TRY(group(&g, 1));
    }

    // ---- modulation and the timestep MLP: Linears of B rows.  Up to
    // kRowsMaxB rows their products run on HBM-bound kernels (the weight
    // gradient is a write of M N fp32, the input gradient a read of the
    // weight); larger batches take the tensor-core GEMM over Kp padded rows.
    const bool few = B <= kRowsMaxB;
    if (few) {
        FF_TRY(rows_wgrad(B, static_cast<int>(Wm), H, p.dmods, Wm, f.tc, H, G("mod.w"), H, stream));
    } else {
        FF_TRY(f32_to_bf16(p.dmods, p.dmods_b, static_cast<int64_t>(B) * Wm, stream));
        if (Kp > B && cudaMemsetAsync(p.dmods_b + static_cast<int64_t>(B) * Wm, 0,
                                      static_cast<size_t>(Kp - B) * Wm * 2, stream) != cudaSuccess)
            return set_error(FF_ERR_CUDA, "backward: memset failed");
        GemmArgs g = wgrad(p.dmods_b, Wm, f.tc, H, static_cast<int>(Wm), H, Kp, G("mod.w"));
        FF_TRY(group(&g, 1));
    }
    FF_TRY(colsum(p.dmods, true, Wm, B, static_cast<int>(Wm), G("mod.b"), p.cs_ws, stream));
    if (few) {
        FF_TRY(rows_dgrad(B, static_cast<int>(Wm), H, p.dmods, Wm, W("mod.w"), H, p.dtc, H, p.rows_part,
                          p.rows_part_floats, stream));
    } else {
        GemmArgs g = dgrad(p.dmods_b, Wm, W("mod.w"), Kp, H, static_cast<int>(Wm));
        g.epi.out_f32 = 1; g.epi.out0 = p.dtc; g.epi.ld0 = H;
        FF_TRY(group(&g, 1));
    }
    FF_TRY(silu_backward(p.dtc, H, f.pre_c, B, Kp, H, p.dc, p.dc_b, stream));
    if (few) {
        FF_TRY(rows_wgrad(B, H, H, p.dc, H, f.th, H, G("t_embed.fc2.w"), H, stream));
    } else {
        GemmArgs g = wgrad(p.dc_b, H, f.th, H, H, H, Kp, G("t_embed.fc2.w"));
        FF_TRY(group(&g, 1));
    }
    FF_TRY(colsum(p.dc, true, H, B, H, G("t_embed.fc2.b"), p.cs_ws, stream));
    if (few) {
        FF_TRY(rows_dgrad(B, H, H, p.dc, H, W("t_embed.fc2.w"), H, p.dth, H, p.rows_part, p.rows_part_floats,
                          stream));
    } else {
        GemmArgs g = dgrad(p.dc_b, H, W("t_embed.fc2.w"), Kp, H, H);
        g.epi.out_f32 = 1; g.epi.out0 = p.dth; g.epi.ld0 = H;
        FF_TRY(group(&g, 1));
    }
    FF_TRY(silu_backward(p.dth, H, f.pre_fc1, B, Kp, H, p.da, p.da_b, stream));
    if (few) {
        FF_TRY(rows_wgrad(B, H, tf, p.da, H, f.temb, tf, G("t_embed.fc1.w"), tf, stream));
    } else {
        GemmArgs g = wgrad(p.da_b, H, f.temb, tf, H, tf, Kp, G("t_embed.fc1.w"));
        FF_TRY(group(&g, 1));
    }
    return colsum(p.da, true, H, B, H, G("t_embed.fc1.b"), p.cs_ws, stream);
}

}  // extern "C"
