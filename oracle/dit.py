"""Velocity v_theta(x_t, t) of a flow-matching MMDiT (fp64).

The paper fixes the role of the network (v_theta in Eq. 1 and Eq. 3) and names
the model families (Flux, Qwen-Image, WAN), but prints no architecture.  The
architecture below is the standard Flux-style MMDiT written out plainly:

  * timestep embedding: 256 sinusoid features of 1000 t (frequencies
    exp(-ln(1e4) j / 128), [cos | sin]), Linear-SiLU-Linear -> c [H];
  * adaLN modulation for every block at once: SiLU(c) W_mod^T + b_mod;
  * patch embedding of the 64-dim latent tokens, text embedding of D_txt;
  * double-stream block (per stream own weights): LN (no affine, eps 1e-6)
    then x (1 + scale) + shift; QKV; per-head RMSNorm of q and k (learned
    scale, eps 1e-6); RoPE over (frame, row, col) axes; attention over the
    joint [text; image] sequence with scale 1/sqrt(d); output projection,
    gated residual; LN-modulate; Linear-GELU(tanh)-Linear; gated residual;
  * single-stream block on the joint sequence: LN-modulate; one Linear to
    [qkv | mlp]; attention as above; one Linear of [attn | GELU(mlp)];
    gated residual;
  * final layer on image tokens: LN-modulate (shift, scale), Linear -> P.

Modulation vector layout (per sample, width L_d 12H + L_s 3H + 2H):
  double block l at l*12H: image (shift1, scale1, gate1, shift2, scale2,
  gate2) then text (same six), each H wide; single block l at L_d*12H + l*3H:
  (shift, scale, gate); final layer last: (shift, scale).

RoPE: the head dim is split into axis slices (a_0, a_1, a_2); within a slice
of width a, the pair (2j, 2j+1) is rotated by pos * theta^(-2j/a).  Text
tokens sit at position (0, 0, 0); image token n of an (F, Hg, Wg) grid at
(n // (Hg Wg), (n // Wg) % Hg, n % Wg).

Parity unpinned as a whole: each piece is pinned in tests/test_oracle_dit.py.
"""
from __future__ import annotations

import math

import numpy as np

LN_EPS = 1e-6
RMS_EPS = 1e-6


# ---------------------------------------------------------------------------
# Parameters
# ---------------------------------------------------------------------------

def mod_width(cfg: dict) -> int:
    H = cfg["hidden"]
    return cfg["n_double"] * 12 * H + cfg["n_single"] * 3 * H + 2 * H


def param_specs(cfg: dict):
    """(name, shape) of every parameter of the MMDiT, in a fixed order."""
    H, F, P, d = cfg["hidden"], cfg["mlp"], cfg["patch_dim"], cfg["head_dim"]
    tf = cfg["time_freq_dim"]
    s = [("t_embed.fc1.w", (H, tf)), ("t_embed.fc1.b", (H,)),
         ("t_embed.fc2.w", (H, H)), ("t_embed.fc2.b", (H,)),
         ("mod.w", (mod_width(cfg), H)), ("mod.b", (mod_width(cfg),)),
         ("img_in.w", (H, P)), ("img_in.b", (H,)),
         ("txt_in.w", (H, cfg["txt_dim"])), ("txt_in.b", (H,))]
    for l in range(cfg["n_double"]):
        for st in ("img", "txt"):
            p = f"double.{l}.{st}."
            s += [(p + "qkv.w", (3 * H, H)), (p + "qkv.b", (3 * H,)),
                  (p + "q_norm.scale", (d,)), (p + "k_norm.scale", (d,)),
                  (p + "proj.w", (H, H)), (p + "proj.b", (H,)),
                  (p + "mlp1.w", (F, H)), (p + "mlp1.b", (F,)),
                  (p + "mlp2.w", (H, F)), (p + "mlp2.b", (H,))]
    for l in range(cfg["n_single"]):
        p = f"single.{l}."
        s += [(p + "linear1.w", (3 * H + F, H)), (p + "linear1.b", (3 * H + F,)),
              (p + "q_norm.scale", (d,)), (p + "k_norm.scale", (d,)),
              (p + "linear2.w", (H, H + F)), (p + "linear2.b", (H,))]
    s += [("final.w", (P, H)), ("final.b", (P,))]
    return s


def widen(bits) -> np.ndarray:
    """Exact float64 value of bf16 bit patterns."""
    b = np.asarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def widen_params(bits_dict: dict) -> dict:
    return {k: widen(v) for k, v in bits_dict.items()}


# ---------------------------------------------------------------------------
# Elementary pieces
# ---------------------------------------------------------------------------

def linear(x, w, b):
    """x W^T + b (nn.Linear convention, W is [out, in])."""
    return x @ w.T + b


def silu(x):
    return x / (1.0 + np.exp(-x))


def gelu_tanh(x):
    """GELU, tanh approximation: x/2 (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))."""
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def layer_norm(x, eps: float = LN_EPS):
    """LayerNorm over the last axis, no affine, population variance."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def modulate(xn, shift, scale):
    return xn * (1.0 + scale) + shift


def rms_norm(x, scale, eps: float = RMS_EPS):
    """RMSNorm over the last axis with a learned scale."""
    ms = (x * x).mean(axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * scale


def timestep_embedding(t, dim: int = 256, max_period: float = 10000.0, factor: float = 1000.0):
    """[B, dim] = [cos(factor t f_j) | sin(factor t f_j)], f_j = max_period^(-j/(dim/2))."""
    half = dim // 2
    freqs = np.exp(-math.log(max_period) * np.arange(half, dtype=np.float64) / half)
    args = factor * np.asarray(t, dtype=np.float64)[:, None] * freqs[None, :]
    return np.concatenate([np.cos(args), np.sin(args)], axis=1)


def image_positions(grid) -> np.ndarray:
    """[N_i, 3] (frame, row, col) of image tokens in row-major grid order."""
    f, h, w = grid
    n = np.arange(f * h * w)
    return np.stack([n // (h * w), (n // w) % h, n % w], axis=1).astype(np.float64)


def rope_angles(pos, axes, theta: float = 10000.0) -> np.ndarray:
    """[N, sum(axes)/2] rotation angles: for axis i of width a, pair j gets
    pos_i * theta^(-2j/a)."""
    pos = np.asarray(pos, dtype=np.float64)
    cols = []
    for i, a in enumerate(axes):
        j = np.arange(a // 2, dtype=np.float64)
        freq = theta ** (-2.0 * j / a)
        cols.append(pos[:, i:i + 1] * freq[None, :])
    return np.concatenate(cols, axis=1)


def apply_rope(x, angles):
    """Rotate interleaved pairs (2p, 2p+1) of x [N, heads, d] by angles [N, d/2]."""
    c = np.cos(angles)[:, None, :]
    s = np.sin(angles)[:, None, :]
    x0 = x[..., 0::2]
    x1 = x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def attention(q, k, v, q_chunk: int = 2048):
    """softmax(q k^T / sqrt(d)) v per head.  q [Nq, h, d]; k, v [Nk, h, d]."""
    nq, nh, d = q.shape
    out = np.empty((nq, nh, v.shape[-1]), dtype=np.float64)
    inv = 1.0 / math.sqrt(d)
    for hh in range(nh):
        kh, vh = k[:, hh, :], v[:, hh, :]
        for q0 in range(0, nq, q_chunk):
            s = (q[q0:q0 + q_chunk, hh, :] @ kh.T) * inv
            s = s - s.max(axis=1, keepdims=True)
            p = np.exp(s)
            p = p / p.sum(axis=1, keepdims=True)
            out[q0:q0 + q_chunk, hh, :] = p @ vh
    return out


def attention_lse(q, k) -> np.ndarray:
    """Per-row log-sum-exp of the scaled scores, natural log: [Nq, h]."""
    nq, nh, d = q.shape
    inv = 1.0 / math.sqrt(d)
    out = np.empty((nq, nh))
    for hh in range(nh):
        s = (q[:, hh, :] @ k[:, hh, :].T) * inv
        m = s.max(axis=1, keepdims=True)
        out[:, hh] = (m + np.log(np.exp(s - m).sum(axis=1, keepdims=True)))[:, 0]
    return out


def attention_backward(q, k, v, dout):
    """Gradients of sum(dout * attention(q, k, v)) w.r.t. q, k and v, written
    out from the definitions: with P = softmax(S), S = q k^T / sqrt(d),
      dV = P^T dO,  dP = dO V^T,  dS = P (dP - rowsum(dP P)),
      dQ = dS K / sqrt(d),  dK = dS^T Q / sqrt(d).
    q, dout [Nq, h, d]; k, v [Nk, h, d]."""
    nq, nh, d = q.shape
    inv = 1.0 / math.sqrt(d)
    dq, dk, dv = np.zeros_like(q, dtype=np.float64), np.zeros_like(k, dtype=np.float64), np.zeros_like(v, dtype=np.float64)
    for hh in range(nh):
        qh, kh, vh, gh = q[:, hh, :], k[:, hh, :], v[:, hh, :], dout[:, hh, :]
        s = (qh @ kh.T) * inv
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=1, keepdims=True)
        dv[:, hh, :] = p.T @ gh
        dp = gh @ vh.T
        ds = p * (dp - (dp * p).sum(axis=1, keepdims=True))
        dq[:, hh, :] = (ds @ kh) * inv
        dk[:, hh, :] = (ds.T @ qh) * inv
    return dq, dk, dv


# ---------------------------------------------------------------------------
# Blocks (one sample at a time: x_* are [N_*, H], mods is [mod_width])
# ---------------------------------------------------------------------------

def _heads(x, nh):
    return x.reshape(x.shape[0], nh, -1)


def double_block(P, l, cfg, x_txt, x_img, mods, ang, rows_txt=None, rows_img=None):
    """One double-stream block.  ang: RoPE angles of the joint [text; image]
    sequence.  rows_*: which output rows to compute (None = all); returns the
    updated residual rows (x_txt[rows_txt], x_img[rows_img])."""
    H, nh = cfg["hidden"], cfg["heads"]
    base = l * 12 * H
    streams = {"img": (x_img, base), "txt": (x_txt, base + 6 * H)}
    q, k, v, m = {}, {}, {}, {}
    for st, (x, off) in streams.items():
        ch = [mods[off + i * H: off + (i + 1) * H] for i in range(6)]
        m[st] = ch
        p = f"double.{l}.{st}."
        h = modulate(layer_norm(x), ch[0], ch[1])
        qkv = linear(h, P[p + "qkv.w"], P[p + "qkv.b"])
        q[st] = rms_norm(_heads(qkv[:, :H], nh), P[p + "q_norm.scale"])
        k[st] = rms_norm(_heads(qkv[:, H:2 * H], nh), P[p + "k_norm.scale"])
        v[st] = _heads(qkv[:, 2 * H:], nh)
    nt = x_txt.shape[0]
    qj = apply_rope(np.concatenate([q["txt"], q["img"]]), ang)
    kj = apply_rope(np.concatenate([k["txt"], k["img"]]), ang)
    vj = np.concatenate([v["txt"], v["img"]])
    rt = np.arange(nt) if rows_txt is None else np.asarray(rows_txt, dtype=np.int64)
    ri = np.arange(x_img.shape[0]) if rows_img is None else np.asarray(rows_img, dtype=np.int64)
    out = {}
    for st, rows, off in (("txt", rt, 0), ("img", ri, nt)):
        x = streams[st][0][rows]
        ch = m[st]
        p = f"double.{l}.{st}."
        o = attention(qj[off + rows], kj, vj).reshape(len(rows), H)
        x = x + ch[2] * linear(o, P[p + "proj.w"], P[p + "proj.b"])
        h = modulate(layer_norm(x), ch[3], ch[4])
        u = gelu_tanh(linear(h, P[p + "mlp1.w"], P[p + "mlp1.b"]))
        x = x + ch[5] * linear(u, P[p + "mlp2.w"], P[p + "mlp2.b"])
        out[st] = x
    return out["txt"], out["img"]


def single_block(P, l, cfg, x, mods, ang, rows=None):
    """One single-stream block on the joint sequence x [N, H]."""
    H, nh = cfg["hidden"], cfg["heads"]
    off = cfg["n_double"] * 12 * H + l * 3 * H
    shift, scale, gate = (mods[off + i * H: off + (i + 1) * H] for i in range(3))
    p = f"single.{l}."
    h = modulate(layer_norm(x), shift, scale)
    y = linear(h, P[p + "linear1.w"], P[p + "linear1.b"])
    q = apply_rope(rms_norm(_heads(y[:, :H], nh), P[p + "q_norm.scale"]), ang)
    k = apply_rope(rms_norm(_heads(y[:, H:2 * H], nh), P[p + "k_norm.scale"]), ang)
    v = _heads(y[:, 2 * H:3 * H], nh)
    r = np.arange(x.shape[0]) if rows is None else np.asarray(rows, dtype=np.int64)
    o = attention(q[r], k, v).reshape(len(r), H)
    cat = np.concatenate([o, gelu_tanh(y[r, 3 * H:])], axis=1)
    return x[r] + gate * linear(cat, P[p + "linear2.w"], P[p + "linear2.b"])


def modulation(P, cfg, t):
    """[B, mod_width]: SiLU(c) W_mod^T + b_mod with c the timestep embedding MLP.

    W_mod is read 12H rows (one double block's share) at a time, so a model
    with many blocks never holds the whole matrix in fp64 at once; every
    output is the same dot product as in one product."""
    emb = timestep_embedding(t, cfg["time_freq_dim"])
    c = linear(silu(linear(emb, P["t_embed.fc1.w"], P["t_embed.fc1.b"])),
               P["t_embed.fc2.w"], P["t_embed.fc2.b"])
    a = silu(c)
    w, b = P["mod.w"], P["mod.b"]
    n = b.shape[0]
    out = np.empty((a.shape[0], n))
    step = 12 * cfg["hidden"]
    for r0 in range(0, n, step):
        out[:, r0:r0 + step] = linear(a, w[r0:r0 + step], b[r0:r0 + step])
    return out


def velocity(P, cfg, x_t, txt, t, img_rows=None):
    """v_theta(x_t, t) of the MMDiT.

    P: {name: float64 array}; x_t [B, N_i, P_dim]; txt [B, N_t, D_txt] (values,
    not bits); t [B].  img_rows: optional index array of image tokens whose
    velocity is wanted (only the last block and the final layer are then
    restricted to those rows).  Returns [B, len(rows), P_dim] float64.
    """
    x_t = np.asarray(x_t, dtype=np.float64)
    txt = np.asarray(txt, dtype=np.float64)
    B = x_t.shape[0]
    H = cfg["hidden"]
    nd, ns = cfg["n_double"], cfg["n_single"]
    mods = modulation(P, cfg, t)
    nt = txt.shape[1]
    pos = np.concatenate([np.zeros((nt, 3)), image_positions(cfg["grid"])])
    ang = rope_angles(pos, cfg["rope_axes"], cfg["rope_theta"])
    n_blocks = nd + ns
    rows = None if img_rows is None else np.asarray(img_rows, dtype=np.int64)
    outs = []
    for b in range(B):
        xi = linear(x_t[b], P["img_in.w"], P["img_in.b"])
        xt = linear(txt[b], P["txt_in.w"], P["txt_in.b"])
        for l in range(nd):
            last = (l == n_blocks - 1) and rows is not None
            if last:
                _, xi = double_block(P, l, cfg, xt, xi, mods[b], ang,
                                     rows_txt=np.zeros(0, np.int64), rows_img=rows)
            else:
                xt, xi = double_block(P, l, cfg, xt, xi, mods[b], ang)
        if ns:
            x = np.concatenate([xt, xi])
            for l in range(ns):
                last = (nd + l == n_blocks - 1) and rows is not None
                if last:
                    xi = single_block(P, l, cfg, x, mods[b], ang, rows=nt + rows)
                    x = None
                else:
                    x = single_block(P, l, cfg, x, mods[b], ang)
            if x is not None:
                xi = x[nt:]
        elif rows is not None and n_blocks == 0:
            xi = xi[rows]
        off = nd * 12 * H + ns * 3 * H
        h = modulate(layer_norm(xi), mods[b, off:off + H], mods[b, off + H:off + 2 * H])
        outs.append(linear(h, P["final.w"], P["final.b"]))
    return np.stack(outs)


# ---------------------------------------------------------------------------
# WAN-style video DiT (self-attention over latent tokens with 3D RoPE,
# cross-attention to the embedded text, gated FFN).  The paper names WAN
# (Sec. 1) without an architecture; the definition below is the one the
# CUDA path implements:
#
#   e  = Linear-SiLU-Linear(sinusoid(1000 t))                      [H]
#   e0 = SiLU(e) W_mod^T + b_mod                                   [6H], shared
#   txt_h = Linear(GELU(Linear(txt)))                              [N_t, H]
#   x = Linear(x_t)                                                [N_i, H]
#   per block l, (shift1, scale1, gate1, shift2, scale2, gate2) = e0 + b_l:
#     h = LN(x) (1 + scale1) + shift1; q, k, v = h W_qkv^T + b
#     q, k <- RoPE(RMSNorm_head(q, k)) over (frame, row, col) axes
#     x += gate1 * (SelfAttn(q, k, v) W_proj^T + b)
#     h = LN(x) * w_cn + b_cn                  (affine LN, no modulation)
#     qc = RMSNorm_head(h W_cq^T + b);  kc, vc = txt_h W_ckv^T + b;
#     kc = RMSNorm_head(kc)                    (no RoPE in cross-attention)
#     x += CrossAttn(qc, kc, vc) W_cproj^T + b (no gate)
#     h = LN(x) (1 + scale2) + shift2
#     x += gate2 * (GELU(h W_1^T + b_1) W_2^T + b_2)
#   final: (shift, scale) = e + b_final (each H), v = (LN(x)(1+scale)+shift) W^T + b
# ---------------------------------------------------------------------------

def wan_param_specs(cfg: dict):
    H, F, P, d = cfg["hidden"], cfg["mlp"], cfg["patch_dim"], cfg["head_dim"]
    tf = cfg["time_freq_dim"]
    s = [("t_embed.fc1.w", (H, tf)), ("t_embed.fc1.b", (H,)),
         ("t_embed.fc2.w", (H, H)), ("t_embed.fc2.b", (H,)),
         ("mod.w", (6 * H, H)), ("mod.b", (6 * H,)),
         ("img_in.w", (H, P)), ("img_in.b", (H,)),
         ("txt_in.w", (H, cfg["txt_dim"])), ("txt_in.b", (H,)),
         ("txt_in2.w", (H, H)), ("txt_in2.b", (H,))]
    for l in range(cfg["n_double"]):
        p = f"blocks.{l}."
        s += [(p + "mod.b", (6 * H,)),
              (p + "qkv.w", (3 * H, H)), (p + "qkv.b", (3 * H,)),
              (p + "q_norm.scale", (d,)), (p + "k_norm.scale", (d,)),
              (p + "proj.w", (H, H)), (p + "proj.b", (H,)),
              (p + "cross_norm.scale", (H,)), (p + "cross_norm.b", (H,)),
              (p + "cross_q.w", (H, H)), (p + "cross_q.b", (H,)), (p + "cross_q_norm.scale", (d,)),
              (p + "cross_kv.w", (2 * H, H)), (p + "cross_kv.b", (2 * H,)), (p + "cross_k_norm.scale", (d,)),
              (p + "cross_proj.w", (H, H)), (p + "cross_proj.b", (H,)),
              (p + "mlp1.w", (F, H)), (p + "mlp1.b", (F,)),
              (p + "mlp2.w", (H, F)), (p + "mlp2.b", (H,))]
    s += [("final.mod.b", (2 * H,)), ("final.w", (P, H)), ("final.b", (P,))]
    return s


def wan_velocity(P, cfg, x_t, txt, t, img_rows=None):
    """v_theta(x_t, t) of the WAN-style DiT.  Same conventions as velocity();
    img_rows restricts the last block and the final layer to those tokens."""
    x_t = np.asarray(x_t, dtype=np.float64)
    txt = np.asarray(txt, dtype=np.float64)
    B = x_t.shape[0]
    H, nh = cfg["hidden"], cfg["heads"]
    L = cfg["n_double"]
    emb = timestep_embedding(t, cfg["time_freq_dim"])
    e = linear(silu(linear(emb, P["t_embed.fc1.w"], P["t_embed.fc1.b"])), P["t_embed.fc2.w"], P["t_embed.fc2.b"])
    e0 = linear(silu(e), P["mod.w"], P["mod.b"])
    ang = rope_angles(image_positions(cfg["grid"]), cfg["rope_axes"], cfg["rope_theta"])
    rows = None if img_rows is None else np.asarray(img_rows, dtype=np.int64)
    outs = []
    for b in range(B):
        th = linear(gelu_tanh(linear(txt[b], P["txt_in.w"], P["txt_in.b"])), P["txt_in2.w"], P["txt_in2.b"])
        x = linear(x_t[b], P["img_in.w"], P["img_in.b"])
        for l in range(L):
            p = f"blocks.{l}."
            m = e0[b] + P[p + "mod.b"]
            sh1, sc1, g1, sh2, sc2, g2 = (m[i * H:(i + 1) * H] for i in range(6))
            h = modulate(layer_norm(x), sh1, sc1)
            qkv = linear(h, P[p + "qkv.w"], P[p + "qkv.b"])
            q = apply_rope(rms_norm(_heads(qkv[:, :H], nh), P[p + "q_norm.scale"]), ang)
            k = apply_rope(rms_norm(_heads(qkv[:, H:2 * H], nh), P[p + "k_norm.scale"]), ang)
            v = _heads(qkv[:, 2 * H:], nh)
            r = np.arange(x.shape[0]) if (rows is None or l < L - 1) else rows
            o = attention(q[r], k, v).reshape(len(r), H)
            x = x[r] + g1 * linear(o, P[p + "proj.w"], P[p + "proj.b"])
            h = layer_norm(x) * P[p + "cross_norm.scale"] + P[p + "cross_norm.b"]
            qc = rms_norm(_heads(linear(h, P[p + "cross_q.w"], P[p + "cross_q.b"]), nh), P[p + "cross_q_norm.scale"])
            kv = linear(th, P[p + "cross_kv.w"], P[p + "cross_kv.b"])
            kc = rms_norm(_heads(kv[:, :H], nh), P[p + "cross_k_norm.scale"])
            vc = _heads(kv[:, H:], nh)
            x = x + linear(attention(qc, kc, vc).reshape(len(r), H), P[p + "cross_proj.w"], P[p + "cross_proj.b"])
            h = modulate(layer_norm(x), sh2, sc2)
            u = gelu_tanh(linear(h, P[p + "mlp1.w"], P[p + "mlp1.b"]))
            x = x + g2 * linear(u, P[p + "mlp2.w"], P[p + "mlp2.b"])
        if L == 0 and rows is not None:
            x = x[rows]
        fm = P["final.mod.b"]
        h = modulate(layer_norm(x), e[b] + fm[:H], e[b] + fm[H:])
        outs.append(linear(h, P["final.w"], P["final.b"]))
    return np.stack(outs)
