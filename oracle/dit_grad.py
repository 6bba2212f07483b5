"""Gradient of the DiT velocity (MMDiT and WAN-style) with respect to its
weights (fp64).

Test infrastructure only (see oracle/__init__.py).  The training half of every
GRPO-style trainer (Sec. 1: forward passes "again for training"; the Flow-GRPO
update of Sec. 3.1, the AWM objective of Eq. 3) differentiates a scalar loss
through v_theta.  Given the loss's gradient dv = dL/dv, ``velocity_vjp``
returns dL/dtheta for every parameter of oracle/dit.py's MMDiT and dL/dx_t
(``wan_velocity_vjp`` the same for the WAN-style network):
the vector-Jacobian product of the velocity, written as the reverse of the
forward in oracle/dit.py, one elementary backward per forward step:

  linear     y = x W^T + b:          dx = dy W, dW = dy^T x, db = sum_rows dy
  layer_norm n = (x - mu) / s:       dx = (dn - mean(dn) - n mean(dn n)) / s
  modulate   y = n (1 + sc) + sh:    dn = dy (1 + sc), dsc = sum dy n, dsh = sum dy
  rms_norm   y = x r w, r = (mean x^2 + eps)^-1/2, xn = x r:
                                     dx = r (g - xn mean(g xn)), g = dy w; dw = sum dy xn
  rope       a rotation per pair:    the transposed rotation (angle negated)
  gelu_tanh  y = x/2 (1 + tanh z), z = k (x + c x^3):
                                     y' = (1 + tanh z)/2 + x/2 (1 - tanh^2 z) k (1 + 3 c x^2)
  silu       y = x sigma(x):         y' = sigma(x) (1 + x (1 - sigma(x)))
  attention                          dit.attention_backward
  gated residual x' = x + g y:       dx += dx', dy = dx' g, dg = sum_rows dx' y

Each elementary backward, and the whole product, is pinned by central
differences (tests/test_oracle_dit_grad.py).  The forward it reverses is
oracle/dit.py's velocity with every row computed (no row restriction).
"""
from __future__ import annotations

import math

import numpy as np

from . import dit

_GELU_K = math.sqrt(2.0 / math.pi)
_GELU_C = 0.044715


# ---------------------------------------------------------------------------
# Elementary backwards
# ---------------------------------------------------------------------------

def linear_bwd(x, w, dy):
    """(dx, dW, db) of y = x W^T + b."""
    return dy @ w, dy.T @ x, dy.sum(axis=0)


def layer_norm_bwd(x, dn, eps: float = dit.LN_EPS):
    """dx of n = layer_norm(x) (no affine) given dn, over the last axis."""
    mu = x.mean(axis=-1, keepdims=True)
    s = np.sqrt(((x - mu) ** 2).mean(axis=-1, keepdims=True) + eps)
    n = (x - mu) / s
    return (dn - dn.mean(axis=-1, keepdims=True) - n * (dn * n).mean(axis=-1, keepdims=True)) / s


def modulate_bwd(n, scale, dy):
    """(dn, dshift, dscale) of y = n (1 + scale) + shift; shift / scale are
    broadcast over rows, so their gradients sum over rows."""
    return dy * (1.0 + scale), dy.sum(axis=0), (dy * n).sum(axis=0)


def rms_norm_bwd(x, w, dy, eps: float = dit.RMS_EPS):
    """(dx, dw) of y = rms_norm(x, w) over the last axis; dw sums over every
    leading axis."""
    r = 1.0 / np.sqrt((x * x).mean(axis=-1, keepdims=True) + eps)
    xn = x * r
    g = dy * w
    dx = r * (g - xn * (g * xn).mean(axis=-1, keepdims=True))
    return dx, (dy * xn).reshape(-1, x.shape[-1]).sum(axis=0)


def rope_bwd(dy, angles):
    """Gradient through dit.apply_rope: the pair rotation transposed."""
    return dit.apply_rope(dy, -angles)


def gelu_tanh_grad(x):
    """d/dx of dit.gelu_tanh."""
    th = np.tanh(_GELU_K * (x + _GELU_C * x ** 3))
    return 0.5 * (1.0 + th) + 0.5 * x * (1.0 - th * th) * _GELU_K * (1.0 + 3.0 * _GELU_C * x * x)


def silu_grad(x):
    """d/dx of dit.silu."""
    s = 1.0 / (1.0 + np.exp(-x))
    return s * (1.0 + x * (1.0 - s))


# ---------------------------------------------------------------------------
# Blocks: forward with the values the backward reads, then the backward
# ---------------------------------------------------------------------------

def _double_fwd(P, l, cfg, x_txt, x_img, mods, ang):
    H, nh = cfg["hidden"], cfg["heads"]
    base = l * 12 * H
    nt = x_txt.shape[0]
    c = {"nt": nt}
    for st, x, off in (("txt", x_txt, base + 6 * H), ("img", x_img, base)):
        p = f"double.{l}.{st}."
        ch = [mods[off + i * H: off + (i + 1) * H] for i in range(6)]
        n1 = dit.layer_norm(x)
        h1 = dit.modulate(n1, ch[0], ch[1])
        qkv = dit.linear(h1, P[p + "qkv.w"], P[p + "qkv.b"])
        qr, kr = dit._heads(qkv[:, :H], nh), dit._heads(qkv[:, H:2 * H], nh)
        c[st] = dict(x=x, ch=ch, off=off, n1=n1, h1=h1, qr=qr, kr=kr,
                     qn=dit.rms_norm(qr, P[p + "q_norm.scale"]),
                     kn=dit.rms_norm(kr, P[p + "k_norm.scale"]),
                     v=dit._heads(qkv[:, 2 * H:], nh))
    q = dit.apply_rope(np.concatenate([c["txt"]["qn"], c["img"]["qn"]]), ang)
    k = dit.apply_rope(np.concatenate([c["txt"]["kn"], c["img"]["kn"]]), ang)
    v = np.concatenate([c["txt"]["v"], c["img"]["v"]])
    o = dit.attention(q, k, v)
    c.update(q=q, k=k, vj=v)
    out = {}
    for st, rows in (("txt", slice(0, nt)), ("img", slice(nt, None))):
        p = f"double.{l}.{st}."
        s = c[st]
        ch = s["ch"]
        s["o"] = o[rows].reshape(-1, H)
        s["y1"] = dit.linear(s["o"], P[p + "proj.w"], P[p + "proj.b"])
        s["x2"] = s["x"] + ch[2] * s["y1"]
        s["n2"] = dit.layer_norm(s["x2"])
        s["h2"] = dit.modulate(s["n2"], ch[3], ch[4])
        s["a"] = dit.linear(s["h2"], P[p + "mlp1.w"], P[p + "mlp1.b"])
        s["u"] = dit.gelu_tanh(s["a"])
        s["y2"] = dit.linear(s["u"], P[p + "mlp2.w"], P[p + "mlp2.b"])
        out[st] = s["x2"] + ch[5] * s["y2"]
    return out["txt"], out["img"], c


def _double_bwd(P, G, l, cfg, c, ang, dx_txt, dx_img, dmods):
    """Accumulates into G (parameter gradients) and dmods; returns the
    gradients of the block's two input residuals."""
    H, nh = cfg["hidden"], cfg["heads"]
    nt = c["nt"]
    dout = {"txt": dx_txt, "img": dx_img}
    do = {}
    for st in ("txt", "img"):
        p = f"double.{l}.{st}."
        s = c[st]
        ch = s["ch"]
        dx3 = dout[st]
        dg2 = (dx3 * s["y2"]).sum(axis=0)
        du, dW, db = linear_bwd(s["u"], P[p + "mlp2.w"], dx3 * ch[5])
        G[p + "mlp2.w"] += dW
        G[p + "mlp2.b"] += db
        da = du * gelu_tanh_grad(s["a"])
        dh2, dW, db = linear_bwd(s["h2"], P[p + "mlp1.w"], da)
        G[p + "mlp1.w"] += dW
        G[p + "mlp1.b"] += db
        dn2, dsh2, dsc2 = modulate_bwd(s["n2"], ch[4], dh2)
        dx2 = dx3 + layer_norm_bwd(s["x2"], dn2)
        dg1 = (dx2 * s["y1"]).sum(axis=0)
        dob, dW, db = linear_bwd(s["o"], P[p + "proj.w"], dx2 * ch[2])
        G[p + "proj.w"] += dW
        G[p + "proj.b"] += db
        do[st] = dob
        s["dx2"] = dx2
        s["dmod"] = [None, None, dg1, dsh2, dsc2, dg2]
    dO = dit._heads(np.concatenate([do["txt"], do["img"]]), nh)
    dq, dk, dv = dit.attention_backward(c["q"], c["k"], c["vj"], dO)
    dqn, dkn = rope_bwd(dq, ang), rope_bwd(dk, ang)
    res = {}
    for st, rows in (("txt", slice(0, nt)), ("img", slice(nt, None))):
        p = f"double.{l}.{st}."
        s = c[st]
        ch = s["ch"]
        dqr, dws = rms_norm_bwd(s["qr"], P[p + "q_norm.scale"], dqn[rows])
        G[p + "q_norm.scale"] += dws
        dkr, dws = rms_norm_bwd(s["kr"], P[p + "k_norm.scale"], dkn[rows])
        G[p + "k_norm.scale"] += dws
        n = dqr.shape[0]
        dqkv = np.concatenate([dqr.reshape(n, H), dkr.reshape(n, H), dv[rows].reshape(n, H)], axis=1)
        dh1, dW, db = linear_bwd(s["h1"], P[p + "qkv.w"], dqkv)
        G[p + "qkv.w"] += dW
        G[p + "qkv.b"] += db
        dn1, dsh1, dsc1 = modulate_bwd(s["n1"], ch[1], dh1)
        res[st] = s["dx2"] + layer_norm_bwd(s["x"], dn1)
        s["dmod"][0], s["dmod"][1] = dsh1, dsc1
        for i in range(6):
            dmods[s["off"] + i * H: s["off"] + (i + 1) * H] += s["dmod"][i]
    return res["txt"], res["img"]


def _single_fwd(P, l, cfg, x, mods, ang):
    H, nh = cfg["hidden"], cfg["heads"]
    off = cfg["n_double"] * 12 * H + l * 3 * H
    p = f"single.{l}."
    ch = [mods[off + i * H: off + (i + 1) * H] for i in range(3)]
    n = dit.layer_norm(x)
    h = dit.modulate(n, ch[0], ch[1])
    y = dit.linear(h, P[p + "linear1.w"], P[p + "linear1.b"])
    qr, kr = dit._heads(y[:, :H], nh), dit._heads(y[:, H:2 * H], nh)
    v = dit._heads(y[:, 2 * H:3 * H], nh)
    q = dit.apply_rope(dit.rms_norm(qr, P[p + "q_norm.scale"]), ang)
    k = dit.apply_rope(dit.rms_norm(kr, P[p + "k_norm.scale"]), ang)
    o = dit.attention(q, k, v).reshape(x.shape[0], H)
    m = y[:, 3 * H:]
    cat = np.concatenate([o, dit.gelu_tanh(m)], axis=1)
    y2 = dit.linear(cat, P[p + "linear2.w"], P[p + "linear2.b"])
    c = dict(x=x, ch=ch, off=off, n=n, h=h, qr=qr, kr=kr, q=q, k=k, v=v, m=m, cat=cat, y2=y2)
    return x + ch[2] * y2, c


def _single_bwd(P, G, l, cfg, c, ang, dout, dmods):
    H, nh = cfg["hidden"], cfg["heads"]
    p = f"single.{l}."
    ch = c["ch"]
    dg = (dout * c["y2"]).sum(axis=0)
    dcat, dW, db = linear_bwd(c["cat"], P[p + "linear2.w"], dout * ch[2])
    G[p + "linear2.w"] += dW
    G[p + "linear2.b"] += db
    dm = dcat[:, H:] * gelu_tanh_grad(c["m"])
    dq, dk, dv = dit.attention_backward(c["q"], c["k"], c["v"], dit._heads(dcat[:, :H], nh))
    dqr, dws = rms_norm_bwd(c["qr"], P[p + "q_norm.scale"], rope_bwd(dq, ang))
    G[p + "q_norm.scale"] += dws
    dkr, dws = rms_norm_bwd(c["kr"], P[p + "k_norm.scale"], rope_bwd(dk, ang))
    G[p + "k_norm.scale"] += dws
    n = dout.shape[0]
    dy = np.concatenate([dqr.reshape(n, H), dkr.reshape(n, H), dv.reshape(n, H), dm], axis=1)
    dh, dW, db = linear_bwd(c["h"], P[p + "linear1.w"], dy)
    G[p + "linear1.w"] += dW
    G[p + "linear1.b"] += db
    dn, dsh, dsc = modulate_bwd(c["n"], ch[1], dh)
    off = c["off"]
    for i, g in enumerate((dsh, dsc, dg)):
        dmods[off + i * H: off + (i + 1) * H] += g
    return dout + layer_norm_bwd(c["x"], dn)


# ---------------------------------------------------------------------------
# The whole network
# ---------------------------------------------------------------------------

def velocity_vjp(P, cfg, x_t, txt, t, dv):
    """v = dit.velocity(P, cfg, x_t, txt, t) and the gradients of
    L = sum(dv * v): (v [B, N_i, P], {name: dL/dP[name]}, dL/dx_t)."""
    x_t = np.asarray(x_t, dtype=np.float64)
    txt = np.asarray(txt, dtype=np.float64)
    dv = np.asarray(dv, dtype=np.float64)
    B = x_t.shape[0]
    H = cfg["hidden"]
    nd, ns = cfg["n_double"], cfg["n_single"]
    G = {k: np.zeros_like(v) for k, v in P.items()}

    # timestep MLP and modulation (batched over samples)
    emb = dit.timestep_embedding(t, cfg["time_freq_dim"])
    a1 = dit.linear(emb, P["t_embed.fc1.w"], P["t_embed.fc1.b"])
    s1 = dit.silu(a1)
    cv = dit.linear(s1, P["t_embed.fc2.w"], P["t_embed.fc2.b"])
    sc = dit.silu(cv)
    mods = dit.linear(sc, P["mod.w"], P["mod.b"])
    dmods = np.zeros_like(mods)

    nt = txt.shape[1]
    pos = np.concatenate([np.zeros((nt, 3)), dit.image_positions(cfg["grid"])])
    ang = dit.rope_angles(pos, cfg["rope_axes"], cfg["rope_theta"])
    off_f = nd * 12 * H + ns * 3 * H
    v_out = []
    dx_t = np.zeros_like(x_t)
    for b in range(B):
        xi = dit.linear(x_t[b], P["img_in.w"], P["img_in.b"])
        xt = dit.linear(txt[b], P["txt_in.w"], P["txt_in.b"])
        caches = []
        for l in range(nd):
            xt, xi, c = _double_fwd(P, l, cfg, xt, xi, mods[b], ang)
            caches.append(c)
        x = np.concatenate([xt, xi])
        for l in range(ns):
            x, c = _single_fwd(P, l, cfg, x, mods[b], ang)
            caches.append(c)
        xi = x[nt:]
        sh, scl = mods[b, off_f:off_f + H], mods[b, off_f + H:off_f + 2 * H]
        nf = dit.layer_norm(xi)
        hf = dit.modulate(nf, sh, scl)
        v_out.append(dit.linear(hf, P["final.w"], P["final.b"]))

        # ---- backward of this sample
        dhf, dW, db = linear_bwd(hf, P["final.w"], dv[b])
        G["final.w"] += dW
        G["final.b"] += db
        dnf, dsh, dsc = modulate_bwd(nf, scl, dhf)
        dmods[b, off_f:off_f + H] += dsh
        dmods[b, off_f + H:off_f + 2 * H] += dsc
        dx = np.concatenate([np.zeros((nt, H)), layer_norm_bwd(xi, dnf)])
        for l in reversed(range(ns)):
            dx = _single_bwd(P, G, l, cfg, caches[nd + l], ang, dx, dmods[b])
        dxt, dxi = dx[:nt], dx[nt:]
        for l in reversed(range(nd)):
            dxt, dxi = _double_bwd(P, G, l, cfg, caches[l], ang, dxt, dxi, dmods[b])
        dxb, dW, db = linear_bwd(x_t[b], P["img_in.w"], dxi)
        G["img_in.w"] += dW
        G["img_in.b"] += db
        dx_t[b] = dxb
        _, dW, db = linear_bwd(txt[b], P["txt_in.w"], dxt)
        G["txt_in.w"] += dW
        G["txt_in.b"] += db

    # modulation and timestep MLP
    dsc_, dW, db = linear_bwd(sc, P["mod.w"], dmods)
    G["mod.w"] += dW
    G["mod.b"] += db
    ds1, dW, db = linear_bwd(s1, P["t_embed.fc2.w"], dsc_ * silu_grad(cv))
    G["t_embed.fc2.w"] += dW
    G["t_embed.fc2.b"] += db
    _, dW, db = linear_bwd(emb, P["t_embed.fc1.w"], ds1 * silu_grad(a1))
    G["t_embed.fc1.w"] += dW
    G["t_embed.fc1.b"] += db
    return np.stack(v_out), G, dx_t


# ---------------------------------------------------------------------------
# The WAN-style network (oracle/dit.py: wan_velocity)
#
# Beyond the MMDiT's steps, its backward needs
#   affine LayerNorm  y = n w + b:      dn = dy w, dw = sum dy n, db = sum dy
#   ungated residual  x' = x + y:       dx += dx', dy = dx'
#   cross-attention   q from the latents, k / v from the embedded text: the
#                     text's gradient sums over every block's k / v products
#   shared modulation block l's vectors are e0 + b_l, the final layer's
#                     e + b_final: d e0 sums over the blocks, d b_l over the
#                     batch, and e collects the final layer's shift and scale
#                     gradients besides the path through SiLU(e)
# ---------------------------------------------------------------------------

def _wan_block_fwd(P, l, cfg, x, th, m, ang):
    H, nh = cfg["hidden"], cfg["heads"]
    p = f"blocks.{l}."
    ch = [m[i * H:(i + 1) * H] for i in range(6)]
    c = dict(x=x, ch=ch)
    c["n1"] = dit.layer_norm(x)
    c["h1"] = dit.modulate(c["n1"], ch[0], ch[1])
    qkv = dit.linear(c["h1"], P[p + "qkv.w"], P[p + "qkv.b"])
    c["qr"], c["kr"] = dit._heads(qkv[:, :H], nh), dit._heads(qkv[:, H:2 * H], nh)
    c["q"] = dit.apply_rope(dit.rms_norm(c["qr"], P[p + "q_norm.scale"]), ang)
    c["k"] = dit.apply_rope(dit.rms_norm(c["kr"], P[p + "k_norm.scale"]), ang)
    c["v"] = dit._heads(qkv[:, 2 * H:], nh)
    c["o"] = dit.attention(c["q"], c["k"], c["v"]).reshape(x.shape[0], H)
    c["y1"] = dit.linear(c["o"], P[p + "proj.w"], P[p + "proj.b"])
    c["x2"] = x + ch[2] * c["y1"]
    c["nc"] = dit.layer_norm(c["x2"])
    c["hc"] = c["nc"] * P[p + "cross_norm.scale"] + P[p + "cross_norm.b"]
    c["qcr"] = dit._heads(dit.linear(c["hc"], P[p + "cross_q.w"], P[p + "cross_q.b"]), nh)
    c["qc"] = dit.rms_norm(c["qcr"], P[p + "cross_q_norm.scale"])
    kv = dit.linear(th, P[p + "cross_kv.w"], P[p + "cross_kv.b"])
    c["kcr"] = dit._heads(kv[:, :H], nh)
    c["kc"] = dit.rms_norm(c["kcr"], P[p + "cross_k_norm.scale"])
    c["vc"] = dit._heads(kv[:, H:], nh)
    c["oc"] = dit.attention(c["qc"], c["kc"], c["vc"]).reshape(x.shape[0], H)
    c["x3"] = c["x2"] + dit.linear(c["oc"], P[p + "cross_proj.w"], P[p + "cross_proj.b"])
    c["n2"] = dit.layer_norm(c["x3"])
    c["h2"] = dit.modulate(c["n2"], ch[3], ch[4])
    c["a"] = dit.linear(c["h2"], P[p + "mlp1.w"], P[p + "mlp1.b"])
    c["u"] = dit.gelu_tanh(c["a"])
    c["y2"] = dit.linear(c["u"], P[p + "mlp2.w"], P[p + "mlp2.b"])
    return c["x3"] + ch[5] * c["y2"], c


def _wan_block_bwd(P, G, l, cfg, c, th, ang, dout, dm, dth):
    """Accumulates the block's parameter gradients into G, its modulation
    vectors' gradient into dm [6H] and the text embedding's into dth; returns
    the gradient of the block's input residual."""
    H, nh = cfg["hidden"], cfg["heads"]
    p = f"blocks.{l}."
    ch = c["ch"]
    n, nt = c["x"].shape[0], th.shape[0]
    # FFN half: x4 = x3 + g2 MLP(LNmod2(x3))
    dm[5 * H:6 * H] += (dout * c["y2"]).sum(axis=0)
    du, dW, db = linear_bwd(c["u"], P[p + "mlp2.w"], dout * ch[5])
    G[p + "mlp2.w"] += dW
    G[p + "mlp2.b"] += db
    dh2, dW, db = linear_bwd(c["h2"], P[p + "mlp1.w"], du * gelu_tanh_grad(c["a"]))
    G[p + "mlp1.w"] += dW
    G[p + "mlp1.b"] += db
    dn2, dsh2, dsc2 = modulate_bwd(c["n2"], ch[4], dh2)
    dm[3 * H:4 * H] += dsh2
    dm[4 * H:5 * H] += dsc2
    dx3 = dout + layer_norm_bwd(c["x3"], dn2)
    # cross-attention half: x3 = x2 + CrossAttn(LN_affine(x2), text)
    doc, dW, db = linear_bwd(c["oc"], P[p + "cross_proj.w"], dx3)
    G[p + "cross_proj.w"] += dW
    G[p + "cross_proj.b"] += db
    dqc, dkc, dvc = dit.attention_backward(c["qc"], c["kc"], c["vc"], dit._heads(doc, nh))
    dqcr, dws = rms_norm_bwd(c["qcr"], P[p + "cross_q_norm.scale"], dqc)
    G[p + "cross_q_norm.scale"] += dws
    dkcr, dws = rms_norm_bwd(c["kcr"], P[p + "cross_k_norm.scale"], dkc)
    G[p + "cross_k_norm.scale"] += dws
    dhc, dW, db = linear_bwd(c["hc"], P[p + "cross_q.w"], dqcr.reshape(n, H))
    G[p + "cross_q.w"] += dW
    G[p + "cross_q.b"] += db
    dkv = np.concatenate([dkcr.reshape(nt, H), dvc.reshape(nt, H)], axis=1)
    dt, dW, db = linear_bwd(th, P[p + "cross_kv.w"], dkv)
    G[p + "cross_kv.w"] += dW
    G[p + "cross_kv.b"] += db
    dth += dt
    G[p + "cross_norm.scale"] += (dhc * c["nc"]).sum(axis=0)
    G[p + "cross_norm.b"] += dhc.sum(axis=0)
    dx2 = dx3 + layer_norm_bwd(c["x2"], dhc * P[p + "cross_norm.scale"])
    # self-attention half: x2 = x + g1 proj(Attn(...))
    dm[2 * H:3 * H] += (dx2 * c["y1"]).sum(axis=0)
    do, dW, db = linear_bwd(c["o"], P[p + "proj.w"], dx2 * ch[2])
    G[p + "proj.w"] += dW
    G[p + "proj.b"] += db
    dq, dk, dv = dit.attention_backward(c["q"], c["k"], c["v"], dit._heads(do, nh))
    dqr, dws = rms_norm_bwd(c["qr"], P[p + "q_norm.scale"], rope_bwd(dq, ang))
    G[p + "q_norm.scale"] += dws
    dkr, dws = rms_norm_bwd(c["kr"], P[p + "k_norm.scale"], rope_bwd(dk, ang))
    G[p + "k_norm.scale"] += dws
    dqkv = np.concatenate([dqr.reshape(n, H), dkr.reshape(n, H), dv.reshape(n, H)], axis=1)
    dh1, dW, db = linear_bwd(c["h1"], P[p + "qkv.w"], dqkv)
    G[p + "qkv.w"] += dW
    G[p + "qkv.b"] += db
    dn1, dsh1, dsc1 = modulate_bwd(c["n1"], ch[1], dh1)
    dm[0:H] += dsh1
    dm[H:2 * H] += dsc1
    return dx2 + layer_norm_bwd(c["x"], dn1)


def wan_velocity_vjp(P, cfg, x_t, txt, t, dv):
    """v = dit.wan_velocity(P, cfg, x_t, txt, t) and the gradients of
    L = sum(dv * v): (v [B, N_i, P], {name: dL/dP[name]}, dL/dx_t)."""
    x_t = np.asarray(x_t, dtype=np.float64)
    txt = np.asarray(txt, dtype=np.float64)
    dv = np.asarray(dv, dtype=np.float64)
    B = x_t.shape[0]
    H, L = cfg["hidden"], cfg["n_double"]
    G = {k: np.zeros_like(v) for k, v in P.items()}

    # timestep embedding e, the shared modulation e0 = SiLU(e) W^T + b
    emb = dit.timestep_embedding(t, cfg["time_freq_dim"])
    a1 = dit.linear(emb, P["t_embed.fc1.w"], P["t_embed.fc1.b"])
    s1 = dit.silu(a1)
    e = dit.linear(s1, P["t_embed.fc2.w"], P["t_embed.fc2.b"])
    se = dit.silu(e)
    e0 = dit.linear(se, P["mod.w"], P["mod.b"])
    de, de0 = np.zeros_like(e), np.zeros_like(e0)
    ang = dit.rope_angles(dit.image_positions(cfg["grid"]), cfg["rope_axes"], cfg["rope_theta"])
    fm = P["final.mod.b"]
    v_out = []
    dx_t = np.zeros_like(x_t)
    for b in range(B):
        at = dit.linear(txt[b], P["txt_in.w"], P["txt_in.b"])
        t1 = dit.gelu_tanh(at)
        th = dit.linear(t1, P["txt_in2.w"], P["txt_in2.b"])
        x = dit.linear(x_t[b], P["img_in.w"], P["img_in.b"])
        caches = []
        for l in range(L):
            x, c = _wan_block_fwd(P, l, cfg, x, th, e0[b] + P[f"blocks.{l}.mod.b"], ang)
            caches.append(c)
        sh, scl = e[b] + fm[:H], e[b] + fm[H:]
        nf = dit.layer_norm(x)
        hf = dit.modulate(nf, sh, scl)
        v_out.append(dit.linear(hf, P["final.w"], P["final.b"]))

        # ---- backward of this sample
        dhf, dW, db = linear_bwd(hf, P["final.w"], dv[b])
        G["final.w"] += dW
        G["final.b"] += db
        dnf, dsh, dsc = modulate_bwd(nf, scl, dhf)
        G["final.mod.b"][:H] += dsh
        G["final.mod.b"][H:] += dsc
        de[b] += dsh + dsc
        dx = layer_norm_bwd(x, dnf)
        dth = np.zeros_like(th)
        for l in reversed(range(L)):
            dm = np.zeros(6 * H)
            dx = _wan_block_bwd(P, G, l, cfg, caches[l], th, ang, dx, dm, dth)
            G[f"blocks.{l}.mod.b"] += dm
            de0[b] += dm
        dxb, dW, db = linear_bwd(x_t[b], P["img_in.w"], dx)
        G["img_in.w"] += dW
        G["img_in.b"] += db
        dx_t[b] = dxb
        dt1, dW, db = linear_bwd(t1, P["txt_in2.w"], dth)
        G["txt_in2.w"] += dW
        G["txt_in2.b"] += db
        _, dW, db = linear_bwd(txt[b], P["txt_in.w"], dt1 * gelu_tanh_grad(at))
        G["txt_in.w"] += dW
        G["txt_in.b"] += db

    # shared modulation and the timestep MLP
    dse, dW, db = linear_bwd(se, P["mod.w"], de0)
    G["mod.w"] += dW
    G["mod.b"] += db
    de += dse * silu_grad(e)
    ds1, dW, db = linear_bwd(s1, P["t_embed.fc2.w"], de)
    G["t_embed.fc2.w"] += dW
    G["t_embed.fc2.b"] += db
    _, dW, db = linear_bwd(emb, P["t_embed.fc1.w"], ds1 * silu_grad(a1))
    G["t_embed.fc1.w"] += dW
    G["t_embed.fc1.b"] += db
    return np.stack(v_out), G, dx_t
