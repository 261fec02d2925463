"""fp64 CPU oracle of the RingAda adapter fine-tuning step (arXiv 2502.19864).

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the cpu-baseline /
reference leg of ``bench.py`` may import or run this module.  It shares no code with the
CUDA path (the package ``paper_2502_19864_gb300``) and imports nothing from it; callers hand
it plain arrays (weights, inputs and labels from ``synth.py``).

What it computes, in the paper's order:
  * Eq. 1 (Section II-A): an adapter maps its input h to h + sigma(h W_down) W_up with
    W_down [n, m], W_up [m, n], no biases.  Two adapters per transformer block (Houlsby
    placement: on the attention-output and FFN-output branches, before the residual add).
  * Algorithm 1, lines "Perform Fw propagation" and "calculates the loss": a forward pass
    through every frozen block, then the head and its cross-entropy loss (Section III-B.2:
    the loss is computed where the labels are).
  * Algorithm 1, line "Perform Bw propagation ending at the (L - d + 1)-th adapter" and
    Section III-B.2: reverse-mode gradients from the loss down to the lowest unfrozen
    layer k = L - d (0-based), giving weight gradients only for the adapters of layers
    >= k and for the head (if trainable), and activation gradients only through layers > k.
    Below k nothing is computed (Section III-A: the clients under the unfreezing depth run
    only the forward).
  * Algorithm 1, "updates the head" and Section III-B.2 "update the parameters of their
    adapter layers": an Adam step on the unfrozen parameters.
  * Algorithm 1, "r mod k = 0 -> d = d + 1": the top-down unfreezing depth schedule.

Readings where the paper is silent (each also listed in the design notes):
  sigma = exact erf GELU; adapters carry no biases; post-LN encoder blocks with LayerNorm
  (biased variance, eps 1e-12) and biased linears; pre-norm decoder blocks with RMSNorm
  (eps 1e-6), causal attention, rotate-half RoPE (theta 10000) and SwiGLU; attention scale
  1/sqrt(head_dim) with no padding mask; encoder head on the token at position 0, or a span
  head (start and end logits at every token, the mean of the two cross-entropies over the
  sequence positions); mean cross-entropy over rows; all gradients, including the one leaving the head, use the
  pre-update weights, and the head and adapters are updated together afterwards; Adam with
  PyTorch's default semantics and a per-parameter step count that starts at the first
  gradient a parameter receives.

Everything is float64.  Weights stored as bf16 arrive as their exact values.
"""
from __future__ import annotations

import numpy as np
from scipy.special import erf

SQRT2 = np.sqrt(2.0)
INV_SQRT_2PI = 1.0 / np.sqrt(2.0 * np.pi)


def f64(a):
    return np.asarray(a, dtype=np.float64)


# ----------------------------------------------------------------------------------------
# Elementwise nonlinearities
# ----------------------------------------------------------------------------------------

def gelu(x):
    """sigma in Eq. 1, read as the exact GELU x * Phi(x)."""
    return 0.5 * x * (1.0 + erf(x / SQRT2))


def gelu_grad(x):
    """d/dx [x Phi(x)] = Phi(x) + x phi(x)."""
    return 0.5 * (1.0 + erf(x / SQRT2)) + x * np.exp(-0.5 * x * x) * INV_SQRT_2PI


def sigmoid(x):
    return 1.0 / (1.0 + np.exp(-x))


def silu(x):
    return x * sigmoid(x)


def silu_grad(x):
    s = sigmoid(x)
    return s * (1.0 + x * (1.0 - s))


# ----------------------------------------------------------------------------------------
# Eq. 1: the adapter and its reverse mode
# ----------------------------------------------------------------------------------------

def adapter_forward(h, W_down, W_up):
    """Eq. 1: h <- h + sigma(h W_down) W_up.  Returns (output, z = h W_down)."""
    z = h @ W_down
    return h + gelu(z) @ W_up, z


def adapter_backward(g, h, z, W_down, W_up, need_dh=True):
    """Gradients of Eq. 1 given g = dLoss/d(output).

    Returns (dh or None, dW_down, dW_up).  dh is skipped at the lowest unfrozen adapter,
    where the backward stops.
    """
    s = gelu(z)
    dW_up = s.T @ g
    dz = (g @ W_up.T) * gelu_grad(z)
    dW_down = h.T @ dz
    dh = (g + dz @ W_down.T) if need_dh else None
    return dh, dW_down, dW_up


# ----------------------------------------------------------------------------------------
# Normalisations
# ----------------------------------------------------------------------------------------

def layer_norm(s, gamma, beta, eps):
    mu = s.mean(axis=-1, keepdims=True)
    var = ((s - mu) ** 2).mean(axis=-1, keepdims=True)
    rstd = 1.0 / np.sqrt(var + eps)
    xhat = (s - mu) * rstd
    return xhat * gamma + beta, (xhat, rstd)


def layer_norm_backward(dy, gamma, cache):
    """dLoss/ds for y = LN(s); gamma and beta are frozen, so only the input gradient."""
    xhat, rstd = cache
    dxhat = dy * gamma
    return rstd * (dxhat - dxhat.mean(axis=-1, keepdims=True)
                   - xhat * (dxhat * xhat).mean(axis=-1, keepdims=True))


def rms_norm(x, gamma, eps):
    r = 1.0 / np.sqrt((x * x).mean(axis=-1, keepdims=True) + eps)
    return x * r * gamma, (x, r)


def rms_norm_backward(dy, gamma, cache):
    x, r = cache
    dn = dy * gamma
    return r * dn - x * (r ** 3) * (dn * x).mean(axis=-1, keepdims=True)


# ----------------------------------------------------------------------------------------
# Attention
# ----------------------------------------------------------------------------------------

def split_heads(t, B, S, n_heads):
    """[B*S, H] -> [B, heads, S, head_dim]."""
    return t.reshape(B, S, n_heads, -1).transpose(0, 2, 1, 3)


def merge_heads(t):
    """[B, heads, S, head_dim] -> [B*S, H]."""
    B, nh, S, dh = t.shape
    return t.transpose(0, 2, 1, 3).reshape(B * S, nh * dh)


def attention(q, k, v, causal):
    """softmax(q k^T / sqrt(dh) [+ causal mask]) v per (batch, head).  Returns (O, P)."""
    dh = q.shape[-1]
    S = q.shape[-2]
    s = (q @ k.transpose(0, 1, 3, 2)) / np.sqrt(dh)
    if causal:
        s = np.where(np.tril(np.ones((S, S), dtype=bool)), s, -np.inf)
    e = np.exp(s - s.max(axis=-1, keepdims=True))
    p = e / e.sum(axis=-1, keepdims=True)
    return p @ v, p


def attention_backward(dO, q, k, v, p):
    dh = q.shape[-1]
    dv = p.transpose(0, 1, 3, 2) @ dO
    dp = dO @ v.transpose(0, 1, 3, 2)
    ds = p * (dp - (dp * p).sum(axis=-1, keepdims=True))
    dq = (ds @ k) / np.sqrt(dh)
    dk = (ds.transpose(0, 1, 3, 2) @ q) / np.sqrt(dh)
    return dq, dk, dv


def rope_tables(S, dh, theta):
    """cos/sin [S, dh/2] for the rotate-half pairing (i, i + dh/2), angle pos*theta^(-2i/dh)."""
    half = dh // 2
    inv_freq = theta ** (-(np.arange(half, dtype=np.float64) * 2.0) / dh)
    ang = np.arange(S, dtype=np.float64)[:, None] * inv_freq[None, :]
    return np.cos(ang), np.sin(ang)


def rope(t, cos, sin):
    half = t.shape[-1] // 2
    t1, t2 = t[..., :half], t[..., half:]
    return np.concatenate([t1 * cos - t2 * sin, t2 * cos + t1 * sin], axis=-1)


def rope_backward(dt, cos, sin):
    """Transpose of the per-pair rotation: rotation by the negative angle."""
    half = dt.shape[-1] // 2
    d1, d2 = dt[..., :half], dt[..., half:]
    return np.concatenate([d1 * cos + d2 * sin, d2 * cos - d1 * sin], axis=-1)


# ----------------------------------------------------------------------------------------
# Loss
# ----------------------------------------------------------------------------------------

def cross_entropy(logits, labels):
    """Mean softmax cross-entropy over rows; returns (loss, dLoss/dlogits)."""
    n = logits.shape[0]
    zmax = logits.max(axis=-1, keepdims=True)
    lse = zmax[:, 0] + np.log(np.exp(logits - zmax).sum(axis=-1))
    loss = float(np.mean(lse - logits[np.arange(n), labels]))
    p = np.exp(logits - lse[:, None])
    p[np.arange(n), labels] -= 1.0
    return loss, p / n


# ----------------------------------------------------------------------------------------
# Transformer blocks with Houlsby adapters
# ----------------------------------------------------------------------------------------

def encoder_layer_forward(x, P, cfg, adapters=True):
    """Post-LN encoder block; adapters on the attention-output and FFN-output branches
    (Houlsby placement), or, with ``cfg.adapters == "paper"``, the single adapter of Fig. 1
    after the FFN add & LayerNorm: out = y2 + sigma(y2 W_down) W_up (Eq. 1 on y2)."""
    B, S, H, nh = cfg.batch, cfg.seq, cfg.hidden, cfg.n_heads
    qkv = x @ P["Wqkv"].T + P["bqkv"]
    q = split_heads(qkv[:, :H], B, S, nh)
    k = split_heads(qkv[:, H:2 * H], B, S, nh)
    v = split_heads(qkv[:, 2 * H:], B, S, nh)
    O, p = attention(q, k, v, causal=False)
    a = merge_heads(O) @ P["Wo"].T + P["bo"]
    if getattr(cfg, "adapters", "houlsby") == "paper":
        y1, ln1 = layer_norm(x + a, P["ln1_g"], P["ln1_b"], cfg.norm_eps)
        u = y1 @ P["W1"].T + P["b1"]
        f = gelu(u) @ P["W2"].T + P["b2"]
        y2, ln2 = layer_norm(y1 + f, P["ln2_g"], P["ln2_b"], cfg.norm_eps)
        if adapters:
            out, zF = adapter_forward(y2, P["WdF"], P["WuF"])
        else:
            out, zF = y2, None
        cache = dict(q=q, k=k, v=v, p=p, ln1=ln1, u=u, y2=y2, zF=zF, ln2=ln2)
        return out, cache
    if adapters:
        a2, zA = adapter_forward(a, P["WdA"], P["WuA"])
    else:
        a2, zA = a, None
    y1, ln1 = layer_norm(x + a2, P["ln1_g"], P["ln1_b"], cfg.norm_eps)
    u = y1 @ P["W1"].T + P["b1"]
    f = gelu(u) @ P["W2"].T + P["b2"]
    if adapters:
        f2, zF = adapter_forward(f, P["WdF"], P["WuF"])
    else:
        f2, zF = f, None
    y2, ln2 = layer_norm(y1 + f2, P["ln2_g"], P["ln2_b"], cfg.norm_eps)
    cache = dict(q=q, k=k, v=v, p=p, a=a, zA=zA, ln1=ln1, u=u, f=f, zF=zF, ln2=ln2)
    return y2, cache


def encoder_layer_backward(dy, P, c, cfg, lowest):
    """Reverse mode through one encoder block.  At the lowest unfrozen layer it stops after
    the attention-branch adapter's weight gradients (no gradient into the block input); with
    the paper's single adapter it stops right after that adapter's weight gradients."""
    grads = {}
    if getattr(cfg, "adapters", "houlsby") == "paper":
        dy2, grads["WdF"], grads["WuF"] = adapter_backward(dy, c["y2"], c["zF"], P["WdF"], P["WuF"],
                                                           need_dh=not lowest)
        if lowest:
            return None, grads
        ds2 = layer_norm_backward(dy2, P["ln2_g"], c["ln2"])
        du = (ds2 @ P["W2"]) * gelu_grad(c["u"])
        dy1 = ds2 + du @ P["W1"]
        ds1 = layer_norm_backward(dy1, P["ln1_g"], c["ln1"])
        dO = split_heads(ds1 @ P["Wo"], cfg.batch, cfg.seq, cfg.n_heads)
        dq, dk, dv = attention_backward(dO, c["q"], c["k"], c["v"], c["p"])
        dqkv = np.concatenate([merge_heads(dq), merge_heads(dk), merge_heads(dv)], axis=1)
        return ds1 + dqkv @ P["Wqkv"], grads
    ds2 = layer_norm_backward(dy, P["ln2_g"], c["ln2"])
    df, grads["WdF"], grads["WuF"] = adapter_backward(ds2, c["f"], c["zF"], P["WdF"], P["WuF"])
    du = (df @ P["W2"]) * gelu_grad(c["u"])
    dy1 = ds2 + du @ P["W1"]
    ds1 = layer_norm_backward(dy1, P["ln1_g"], c["ln1"])
    da, grads["WdA"], grads["WuA"] = adapter_backward(
        ds1, c["a"], c["zA"], P["WdA"], P["WuA"], need_dh=not lowest)
    if lowest:
        return None, grads
    dO = split_heads(da @ P["Wo"], cfg.batch, cfg.seq, cfg.n_heads)
    dq, dk, dv = attention_backward(dO, c["q"], c["k"], c["v"], c["p"])
    dqkv = np.concatenate([merge_heads(dq), merge_heads(dk), merge_heads(dv)], axis=1)
    return ds1 + dqkv @ P["Wqkv"], grads


def decoder_layer_forward(x, P, cfg, rope_cs, adapters=True):
    """Pre-RMSNorm decoder block: causal RoPE attention and SwiGLU FFN, with an adapter on
    each branch before its residual add."""
    B, S, nh = cfg.batch, cfg.seq, cfg.n_heads
    cos, sin = rope_cs
    n1, rms1 = rms_norm(x, P["rms1_g"], cfg.norm_eps)
    q = rope(split_heads(n1 @ P["Wq"].T, B, S, nh), cos, sin)
    k = rope(split_heads(n1 @ P["Wk"].T, B, S, nh), cos, sin)
    v = split_heads(n1 @ P["Wv"].T, B, S, nh)
    O, p = attention(q, k, v, causal=True)
    a = merge_heads(O) @ P["Wo"].T
    if adapters:
        a2, zA = adapter_forward(a, P["WdA"], P["WuA"])
    else:
        a2, zA = a, None
    x1 = x + a2
    n2, rms2 = rms_norm(x1, P["rms2_g"], cfg.norm_eps)
    gate = n2 @ P["Wg"].T
    up = n2 @ P["Wu"].T
    f = (silu(gate) * up) @ P["Wd"].T
    if adapters:
        f2, zF = adapter_forward(f, P["WdF"], P["WuF"])
    else:
        f2, zF = f, None
    cache = dict(rms1=rms1, q=q, k=k, v=v, p=p, a=a, zA=zA, rms2=rms2, gate=gate, up=up,
                 f=f, zF=zF)
    return x1 + f2, cache


def decoder_layer_backward(dx2, P, c, cfg, rope_cs, lowest):
    cos, sin = rope_cs
    grads = {}
    df, grads["WdF"], grads["WuF"] = adapter_backward(dx2, c["f"], c["zF"], P["WdF"], P["WuF"])
    dh = df @ P["Wd"]
    dgate = dh * c["up"] * silu_grad(c["gate"])
    dup = dh * silu(c["gate"])
    dn2 = dgate @ P["Wg"] + dup @ P["Wu"]
    dx1 = dx2 + rms_norm_backward(dn2, P["rms2_g"], c["rms2"])
    da, grads["WdA"], grads["WuA"] = adapter_backward(
        dx1, c["a"], c["zA"], P["WdA"], P["WuA"], need_dh=not lowest)
    if lowest:
        return None, grads
    dO = split_heads(da @ P["Wo"], cfg.batch, cfg.seq, cfg.n_heads)
    dq, dk, dv = attention_backward(dO, c["q"], c["k"], c["v"], c["p"])
    dq = merge_heads(rope_backward(dq, cos, sin))
    dk = merge_heads(rope_backward(dk, cos, sin))
    dv = merge_heads(dv)
    dn1 = dq @ P["Wq"] + dk @ P["Wk"] + dv @ P["Wv"]
    return dx1 + rms_norm_backward(dn1, P["rms1_g"], c["rms1"]), grads


# ----------------------------------------------------------------------------------------
# Heads (Hed)
# ----------------------------------------------------------------------------------------

def encoder_head(y, head, labels, cfg):
    """CLS (position 0) linear head + mean cross-entropy.  Returns loss, logits, dy, grads."""
    B, S, H = cfg.batch, cfg.seq, cfg.hidden
    cls = y.reshape(B, S, H)[:, 0, :]
    logits = cls @ head["Wh"].T + head["bh"]
    loss, dlogits = cross_entropy(logits, labels)
    dy = np.zeros((B, S, H))
    dy[:, 0, :] = dlogits @ head["Wh"]
    grads = dict(Wh=dlogits.T @ cls, bh=dlogits.sum(axis=0))
    return loss, logits, dy.reshape(B * S, H), grads


def encoder_span_head(y, head, labels, cfg):
    """Span head of extractive question answering (the paper's SQuAD task, Section IV):
    start and end logits at every token, [B, S, 2] = y Wh^T + bh with Wh [2, H]; the loss is
    the mean of the start and end cross-entropies, each a softmax over the S positions of a
    sequence, averaged over the batch.  labels [B, 2] = (start, end).  Returns loss, logits
    [B*S, 2], dy [B*S, H] (every position receives a gradient) and the head gradients."""
    B, S, H = cfg.batch, cfg.seq, cfg.hidden
    labels = np.asarray(labels).reshape(B, 2)
    logits = y @ head["Wh"].T + head["bh"]                      # [B*S, 2]
    z = logits.reshape(B, S, 2)
    loss_start, d_start = cross_entropy(z[:, :, 0], labels[:, 0])
    loss_end, d_end = cross_entropy(z[:, :, 1], labels[:, 1])
    loss = 0.5 * (loss_start + loss_end)
    dlogits = 0.5 * np.stack([d_start, d_end], axis=-1).reshape(B * S, 2)
    dy = dlogits @ head["Wh"]
    grads = dict(Wh=dlogits.T @ y, bh=dlogits.sum(axis=0))
    return loss, logits, dy, grads


def decoder_head(y, head, labels, cfg):
    """Final RMSNorm, frozen vocabulary projection, mean next-token cross-entropy over
    all B*S positions (label[b, t] is the target at position t)."""
    n, cache = rms_norm(y, head["rmsf_g"], cfg.norm_eps)
    logits = n @ head["Wh"].T
    loss, dlogits = cross_entropy(logits, labels.reshape(-1))
    dy = rms_norm_backward(dlogits @ head["Wh"], head["rmsf_g"], cache)
    return loss, logits, dy, {}


# ----------------------------------------------------------------------------------------
# The step: forward, loss, early-stopped backward (Algorithm 1)
# ----------------------------------------------------------------------------------------

def to_f64_params(layers, head):
    return [{k: f64(v) for k, v in p.items()} for p in layers], {k: f64(v) for k, v in head.items()}


def forward(cfg, layers, head, x, labels, d, adapters=True, start_layer=0, h0=None):
    """Forward through all layers and the loss.  Caches are kept only for layers >= k.

    ``start_layer``/``h0`` let a caller resume from a known block input (used to make
    finite differences on the top layers cheap); by default the forward starts at x.
    """
    L = cfg.n_layers
    k = L - d
    T, H = cfg.tokens, cfg.hidden
    h = f64(x).reshape(T, H) if h0 is None else f64(h0)
    rope_cs = rope_tables(cfg.seq, cfg.head_dim, cfg.rope_theta) if cfg.arch == "decoder" else None
    caches = {}
    inputs = {}
    for l in range(start_layer, L):
        inputs[l] = h
        if cfg.arch == "encoder":
            h, c = encoder_layer_forward(h, layers[l], cfg, adapters)
        else:
            h, c = decoder_layer_forward(h, layers[l], cfg, rope_cs, adapters)
        if l >= k:
            caches[l] = c
    labels = np.asarray(labels).astype(np.int64)
    if cfg.arch == "encoder" and getattr(cfg, "head", "cls") == "span":
        loss, logits, dy, hgrads = encoder_span_head(h, head, labels, cfg)
    elif cfg.arch == "encoder":
        loss, logits, dy, hgrads = encoder_head(h, head, labels, cfg)
    else:
        loss, logits, dy, hgrads = decoder_head(h, head, labels, cfg)
    return dict(loss=loss, logits=logits, y=h, dy=dy, head_grads=hgrads, caches=caches,
                inputs=inputs, k=k, rope_cs=rope_cs)


def backward_truncated(cfg, layers, fwd, k):
    """Reverse mode from the loss down to layer k, stopping there (Algorithm 1).

    Returns {layer: {WdA, WuA, WdF, WuF}} for layers k..L-1 only, and the gradient that
    enters each block's output (for the layers that were traversed).
    """
    L = cfg.n_layers
    if k < fwd["k"]:
        raise ValueError("layers below the forward's depth were not cached")
    dy = fwd["dy"]
    grads = {}
    dys = {}
    for l in range(L - 1, k - 1, -1):
        dys[l] = dy
        if cfg.arch == "encoder":
            dy, grads[l] = encoder_layer_backward(dy, layers[l], fwd["caches"][l], cfg, l == k)
        else:
            dy, grads[l] = decoder_layer_backward(dy, layers[l], fwd["caches"][l], cfg,
                                                  fwd["rope_cs"], l == k)
    return grads, dys


def step(cfg, layers, head, x, labels, d):
    """One step's forward, loss and early-stopped backward at depth d (k = L - d)."""
    fwd = forward(cfg, layers, head, x, labels, d)
    grads, _ = backward_truncated(cfg, layers, fwd, cfg.n_layers - d)
    head_grads = fwd["head_grads"] if cfg.head_trainable else {}
    return dict(loss=fwd["loss"], logits=fwd["logits"], y=fwd["y"], grads=grads,
                head_grads=head_grads, k=cfg.n_layers - d)


# ----------------------------------------------------------------------------------------
# Update and schedule
# ----------------------------------------------------------------------------------------

class Adam:
    """Adam (PyTorch default semantics, no weight decay) over named parameters.

    A parameter's step count starts at its first gradient, so an adapter unfrozen late
    starts at t = 1 with zero moments.
    """

    def __init__(self, lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8):
        self.lr, self.beta1, self.beta2, self.eps = lr, beta1, beta2, eps
        self.state = {}

    def update(self, name, param, grad):
        m, v, t = self.state.get(name, (np.zeros_like(param), np.zeros_like(param), 0))
        t += 1
        m = self.beta1 * m + (1.0 - self.beta1) * grad
        v = self.beta2 * v + (1.0 - self.beta2) * grad * grad
        bc1 = 1.0 - self.beta1 ** t
        bc2 = 1.0 - self.beta2 ** t
        denom = np.sqrt(v) / np.sqrt(bc2) + self.eps
        self.state[name] = (m, v, t)
        return param - (self.lr / bc1) * m / denom


def apply_update(cfg, layers, head, result, opt):
    """Algorithm 1 "updates the head" and Section III-B.2 adapter updates, applied together
    after the backward (all gradients used the pre-update weights)."""
    for l, g in result["grads"].items():
        for key, gk in g.items():
            layers[l][key] = opt.update((l, key), layers[l][key], gk)
    for key, gk in result["head_grads"].items():
        head[key] = opt.update(("head", key), head[key], gk)


def unfreezing_depth(step_index, interval, d0, d_max):
    """Algorithm 1's top-down schedule with a per-step interval: d grows by one each time
    ``interval`` steps have completed, from d0, capped at d_max."""
    return min(d0 + step_index // interval, d_max)


def train(cfg, layers, head, batches, depths, opt):
    """Run consecutive steps; ``batches`` is a list of (x, labels), ``depths`` the depth
    per step.  Parameters are updated in place; returns the losses."""
    losses = []
    for (x, labels), d in zip(batches, depths):
        r = step(cfg, layers, head, x, labels, d)
        apply_update(cfg, layers, head, r, opt)
        losses.append(r["loss"])
    return losses
