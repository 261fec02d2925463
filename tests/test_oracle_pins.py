"""Pins for the fp64 oracle, independent of the oracle's own code.

Each test checks the oracle against something the paper or mathematics fixes: textbook
values, a library routine that implements the same definition (torch fp64 on the CPU),
closed forms and invariants, central finite differences, and the paper's own worked
example of the early-stopped backward (Fig. 2).  None of these calls the CUDA path.
"""
import json
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as Fnn

import synth
from oracle import ringada_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def T(a, grad=False):
    t = torch.tensor(np.asarray(a, dtype=np.float64), dtype=torch.float64)
    return t.requires_grad_(grad)


def rng(seed=0):
    return np.random.default_rng(seed)


# ----------------------------------------------------------------------------------------
# elementwise pieces
# ----------------------------------------------------------------------------------------

def test_gelu_textbook_values():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "normal_cdf.txt"))
            if l.strip() and not l.startswith("#")]
    for xs, phis in rows:
        x, phi = float(xs), float(phis)
        assert O.gelu(np.array(x)) == pytest.approx(x * phi, rel=1e-14, abs=1e-300)


def test_gelu_and_derivative_match_torch():
    x = rng().normal(size=1000) * 3
    xt = T(x, True)
    y = Fnn.gelu(xt, approximate="none")
    y.sum().backward()
    np.testing.assert_allclose(O.gelu(x), y.detach().numpy(), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(O.gelu_grad(x), xt.grad.numpy(), rtol=1e-13, atol=1e-15)


def test_silu_matches_torch():
    x = rng(1).normal(size=500) * 4
    xt = T(x, True)
    Fnn.silu(xt).sum().backward()
    np.testing.assert_allclose(O.silu(x), Fnn.silu(T(x)).numpy(), rtol=1e-14)
    np.testing.assert_allclose(O.silu_grad(x), xt.grad.numpy(), rtol=1e-13, atol=1e-15)


# ----------------------------------------------------------------------------------------
# norms
# ----------------------------------------------------------------------------------------

def test_layer_norm_matches_torch_and_backward_invariants():
    r = rng(2)
    s = r.normal(size=(7, 96)) * 2 + 0.3
    g = 1 + 0.1 * r.normal(size=96)
    b = 0.1 * r.normal(size=96)
    dy = r.normal(size=(7, 96))
    st = T(s, True)
    y = Fnn.layer_norm(st, (96,), T(g), T(b), eps=1e-12)
    (y * T(dy)).sum().backward()
    yo, cache = O.layer_norm(s, g, b, 1e-12)
    np.testing.assert_allclose(yo, y.detach().numpy(), rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(O.layer_norm_backward(dy, g, cache), st.grad.numpy(),
                               rtol=1e-10, atol=1e-12)
    # closed forms with gamma = 1: the input gradient is orthogonal to 1 and to xhat
    ds = O.layer_norm_backward(dy, np.ones(96), cache)
    xhat = cache[0]
    assert np.abs(ds.sum(-1)).max() < 1e-12
    assert np.abs((ds * xhat).sum(-1)).max() < 1e-11


def test_rms_norm_matches_torch():
    r = rng(3)
    x = r.normal(size=(5, 64))
    g = 1 + 0.1 * r.normal(size=64)
    dy = r.normal(size=(5, 64))
    xt = T(x, True)
    y = Fnn.rms_norm(xt, (64,), T(g), eps=1e-6)
    (y * T(dy)).sum().backward()
    yo, cache = O.rms_norm(x, g, 1e-6)
    np.testing.assert_allclose(yo, y.detach().numpy(), rtol=1e-13)
    np.testing.assert_allclose(O.rms_norm_backward(dy, g, cache), xt.grad.numpy(),
                               rtol=1e-11, atol=1e-13)


# ----------------------------------------------------------------------------------------
# attention, RoPE, cross-entropy
# ----------------------------------------------------------------------------------------

@pytest.mark.parametrize("causal", [False, True])
def test_attention_matches_sdpa(causal):
    r = rng(4)
    q, k, v, do = (r.normal(size=(2, 3, 17, 8)) for _ in range(4))
    qt, kt, vt = T(q, True), T(k, True), T(v, True)
    o = Fnn.scaled_dot_product_attention(qt, kt, vt, is_causal=causal)
    (o * T(do)).sum().backward()
    oo, p = O.attention(q, k, v, causal)
    np.testing.assert_allclose(oo, o.detach().numpy(), rtol=1e-12, atol=1e-13)
    dq, dk, dv = O.attention_backward(do, q, k, v, p)
    np.testing.assert_allclose(dq, qt.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dk, kt.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dv, vt.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_attention_special_cases():
    r = rng(5)
    # one key: softmax of a single score is 1, so O = V
    q, k, v = (r.normal(size=(2, 2, 1, 4)) for _ in range(3))
    np.testing.assert_array_equal(O.attention(q, k, v, False)[0], v)
    # zero queries: uniform weights, O = mean of V over keys
    q = np.zeros((1, 2, 6, 4))
    k, v = r.normal(size=(1, 2, 6, 4)), r.normal(size=(1, 2, 6, 4))
    np.testing.assert_allclose(O.attention(q, k, v, False)[0],
                               np.broadcast_to(v.mean(axis=2, keepdims=True), v.shape), rtol=1e-14)
    # causal: the first query sees only the first key
    q, k, v = (r.normal(size=(1, 1, 5, 4)) for _ in range(3))
    np.testing.assert_allclose(O.attention(q, k, v, True)[0][0, 0, 0], v[0, 0, 0], rtol=1e-15)


def test_rope_properties():
    r = rng(6)
    S, dh = 12, 8
    cos, sin = O.rope_tables(S, dh, 10000.0)
    x = r.normal(size=(1, 1, S, dh))
    y = r.normal(size=(1, 1, S, dh))
    rx = O.rope(x, cos, sin)
    # position 0 is not rotated
    np.testing.assert_array_equal(rx[..., 0, :], x[..., 0, :])
    # a rotation per pair preserves each token's norm
    np.testing.assert_allclose(np.linalg.norm(rx, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-14)
    # the backward is the transpose of the forward map
    assert np.sum(rx * y) == pytest.approx(np.sum(x * O.rope_backward(y, cos, sin)), rel=1e-13)
    # q.k after RoPE depends on the relative position only
    q1, k1 = r.normal(size=dh), r.normal(size=dh)
    Q = np.zeros((1, 1, S, dh)); K = np.zeros((1, 1, S, dh))
    Q[..., :, :] = q1; K[..., :, :] = k1
    rq, rk = O.rope(Q, cos, sin)[0, 0], O.rope(K, cos, sin)[0, 0]
    assert rq[5] @ rk[2] == pytest.approx(rq[9] @ rk[6], rel=1e-12)
    assert rq[3] @ rk[3] == pytest.approx(q1 @ k1, rel=1e-12)
    # frequencies of the rotate-half pairing: pair i turns by theta^(-2i/dh) per position
    assert cos[1, 1] == pytest.approx(np.cos(10000.0 ** (-2.0 / dh)), rel=1e-15)


def test_cross_entropy_matches_torch():
    r = rng(7)
    z = r.normal(size=(9, 13)) * 3
    y = r.integers(0, 13, size=9)
    zt = T(z, True)
    l = Fnn.cross_entropy(zt, torch.tensor(y))
    l.backward()
    loss, dz = O.cross_entropy(z, y)
    assert loss == pytest.approx(l.item(), rel=1e-14)
    np.testing.assert_allclose(dz, zt.grad.numpy(), rtol=1e-12, atol=1e-15)
    assert np.abs(dz.sum(axis=1)).max() < 1e-15
    # equal logits: the loss is ln C
    assert O.cross_entropy(np.zeros((3, 5)), np.array([0, 1, 4]))[0] == pytest.approx(np.log(5), rel=1e-15)


def test_span_head_matches_torch_autograd():
    """Span head (start/end logits at every token): loss, the gradient into every token and
    the head gradients against torch's cross_entropy over the sequence positions."""
    import dataclasses
    cfg = dataclasses.replace(synth.CONFIGS["tiny_span"], batch=3, seq=11, hidden=16)
    r = rng(12)
    y = r.normal(size=(cfg.batch * cfg.seq, cfg.hidden))
    head = dict(Wh=r.normal(size=(2, cfg.hidden)) * 0.3, bh=r.normal(size=2))
    labels = r.integers(0, cfg.seq, size=(cfg.batch, 2))
    loss, logits, dy, g = O.encoder_span_head(y, head, labels, cfg)
    yt, Wt, bt = T(y, True), T(head["Wh"], True), T(head["bh"], True)
    z = (yt @ Wt.T + bt).reshape(cfg.batch, cfg.seq, 2)
    lab = torch.tensor(labels)
    lt = 0.5 * (Fnn.cross_entropy(z[:, :, 0], lab[:, 0]) + Fnn.cross_entropy(z[:, :, 1], lab[:, 1]))
    lt.backward()
    assert loss == pytest.approx(lt.item(), rel=1e-14)
    np.testing.assert_allclose(logits, z.detach().reshape(-1, 2).numpy(), rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(dy, yt.grad.numpy(), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(g["Wh"], Wt.grad.numpy(), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(g["bh"], bt.grad.numpy(), rtol=1e-12, atol=1e-15)
    # each sequence's start (and end) gradients sum to zero over its positions
    d = dy @ np.linalg.pinv(head["Wh"])
    assert np.abs(d.reshape(cfg.batch, cfg.seq, 2).sum(axis=1)).max() < 1e-12
    # equal logits everywhere: the loss is ln S
    flat = dict(Wh=np.zeros((2, cfg.hidden)), bh=np.zeros(2))
    assert O.encoder_span_head(y, flat, labels, cfg)[0] == pytest.approx(np.log(cfg.seq), rel=1e-15)


# ----------------------------------------------------------------------------------------
# adapter (Eq. 1)
# ----------------------------------------------------------------------------------------

def test_adapter_eq1_and_zero_up_projection():
    r = rng(8)
    h = r.normal(size=(11, 32))
    Wd, Wu = r.normal(size=(32, 4)) * 0.1, r.normal(size=(4, 32)) * 0.1
    out, z = O.adapter_forward(h, Wd, Wu)
    # Eq. 1 with sigma = GELU, written with torch's own GELU and matmul
    ref = T(h) + Fnn.gelu(T(h) @ T(Wd)) @ T(Wu)
    np.testing.assert_allclose(out, ref.numpy(), rtol=1e-14, atol=1e-15)
    # W_up = 0: the adapter is the identity, bitwise, and W_down receives no gradient
    out0, z0 = O.adapter_forward(h, Wd, np.zeros_like(Wu))
    np.testing.assert_array_equal(out0, h)
    g = r.normal(size=h.shape)
    dh, dWd, dWu = O.adapter_backward(g, h, z0, Wd, np.zeros_like(Wu))
    np.testing.assert_array_equal(dWd, 0.0)
    np.testing.assert_array_equal(dh, g)
    assert np.abs(dWu).max() > 0


# ----------------------------------------------------------------------------------------
# whole encoder block against torch.nn.TransformerEncoderLayer
# ----------------------------------------------------------------------------------------

class _AttnWithAdapter(torch.nn.Module):
    def __init__(self, mha, Wd, Wu):
        super().__init__()
        self.mha = mha
        self.Wd = torch.nn.Parameter(T(Wd))
        self.Wu = torch.nn.Parameter(T(Wu))

    def forward(self, q, k, v, **kw):
        out, w = self.mha(q, k, v, **kw)
        return out + Fnn.gelu(out @ self.Wd) @ self.Wu, w


class _LinearWithAdapter(torch.nn.Module):
    def __init__(self, lin, Wd, Wu):
        super().__init__()
        self.lin = lin
        self.Wd = torch.nn.Parameter(T(Wd))
        self.Wu = torch.nn.Parameter(T(Wu))

    def forward(self, x):
        f = self.lin(x)
        return f + Fnn.gelu(f @ self.Wd) @ self.Wu


def _torch_encoder_layer(cfg, P, adapters=True):
    H = cfg.hidden
    lay = torch.nn.TransformerEncoderLayer(H, cfg.n_heads, cfg.ffn, dropout=0.0,
                                           activation="gelu", layer_norm_eps=cfg.norm_eps,
                                           batch_first=True, norm_first=False,
                                           dtype=torch.float64)
    with torch.no_grad():
        lay.self_attn.in_proj_weight.copy_(T(P["Wqkv"]))
        lay.self_attn.in_proj_bias.copy_(T(P["bqkv"]))
        lay.self_attn.out_proj.weight.copy_(T(P["Wo"]))
        lay.self_attn.out_proj.bias.copy_(T(P["bo"]))
        lay.linear1.weight.copy_(T(P["W1"])); lay.linear1.bias.copy_(T(P["b1"]))
        lay.linear2.weight.copy_(T(P["W2"])); lay.linear2.bias.copy_(T(P["b2"]))
        lay.norm1.weight.copy_(T(P["ln1_g"])); lay.norm1.bias.copy_(T(P["ln1_b"]))
        lay.norm2.weight.copy_(T(P["ln2_g"])); lay.norm2.bias.copy_(T(P["ln2_b"]))
    for p in lay.parameters():
        p.requires_grad_(False)
    if adapters:
        lay.self_attn = _AttnWithAdapter(lay.self_attn, P["WdA"], P["WuA"])
        lay.linear2 = _LinearWithAdapter(lay.linear2, P["WdF"], P["WuF"])
    lay.train()   # dropout is 0; training mode keeps torch off its fused inference path
    return lay


def _small_enc_cfg():
    return synth.ModelCfg("encoder", 3, 48, 4, 96, 6, 3, 3, 10, "f32")


def _stress_workload(cfg, seed=0, up_std=0.05):
    """The synthetic recipe with a larger adapter up-projection, so that every gradient
    is well above rounding noise in the checks below."""
    w = synth.make_workload(cfg, seed)
    r = rng(100 + seed)
    for p in w["layers"]:
        for key in ("WuA", "WuF"):
            if key in p:
                p[key] = r.normal(size=p[key].shape) * up_std
    return w


def test_encoder_stack_matches_torch_layers_with_autograd():
    """Forward, loss and every adapter/head gradient at full depth against a model built
    from torch's own TransformerEncoderLayer (adapters inserted by wrapping its attention
    and second linear), differentiated by autograd."""
    cfg = _small_enc_cfg()
    w = _stress_workload(cfg)
    layers, head = O.to_f64_params(w["layers"], w["head"])
    res = O.step(cfg, layers, head, w["x"], w["labels"], cfg.n_layers)

    mods = [_torch_encoder_layer(cfg, P) for P in layers]
    Wh, bh = T(head["Wh"], True), T(head["bh"], True)
    h = T(w["x"])
    for m in mods:
        h = m(h)
    logits = h[:, 0, :] @ Wh.T + bh
    loss = Fnn.cross_entropy(logits, torch.tensor(w["labels"]).long())
    loss.backward()
    assert res["loss"] == pytest.approx(loss.item(), rel=1e-12)
    np.testing.assert_allclose(res["logits"], logits.detach().numpy(), rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(res["head_grads"]["Wh"], Wh.grad.numpy(), rtol=1e-9, atol=1e-14)
    np.testing.assert_allclose(res["head_grads"]["bh"], bh.grad.numpy(), rtol=1e-9, atol=1e-14)
    for l, m in enumerate(mods):
        pairs = dict(WdA=m.self_attn.Wd, WuA=m.self_attn.Wu, WdF=m.linear2.Wd, WuF=m.linear2.Wu)
        for key, par in pairs.items():
            g = par.grad.numpy()
            err = np.linalg.norm(res["grads"][l][key] - g) / np.linalg.norm(g)
            assert err < 1e-10, (l, key, err)


def test_paper_placement_matches_torch_layers_with_autograd():
    """The paper's single adapter per block (Fig. 1, after the FFN add & LayerNorm): torch's
    TransformerEncoderLayer without adapters, followed by Eq. 1 on its output, under
    autograd; and the early-stopped backward equals the full one above k, bitwise."""
    import dataclasses
    cfg = dataclasses.replace(_small_enc_cfg(), adapters="paper")
    w = _stress_workload(cfg)
    layers, head = O.to_f64_params(w["layers"], w["head"])
    res = O.step(cfg, layers, head, w["x"], w["labels"], cfg.n_layers)
    mods = [_torch_encoder_layer(cfg, P, adapters=False) for P in layers]
    ad = [(T(P["WdF"], True), T(P["WuF"], True)) for P in layers]
    Wh, bh = T(head["Wh"], True), T(head["bh"], True)
    h = T(w["x"])
    for m, (Wd, Wu) in zip(mods, ad):
        y = m(h)
        h = y + Fnn.gelu(y @ Wd) @ Wu
    logits = h[:, 0, :] @ Wh.T + bh
    loss = Fnn.cross_entropy(logits, torch.tensor(w["labels"]).long())
    loss.backward()
    assert res["loss"] == pytest.approx(loss.item(), rel=1e-12)
    np.testing.assert_allclose(res["logits"], logits.detach().numpy(), rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(res["head_grads"]["Wh"], Wh.grad.numpy(), rtol=1e-9, atol=1e-14)
    for l, (Wd, Wu) in enumerate(ad):
        assert sorted(res["grads"][l]) == ["WdF", "WuF"]
        for key, par in (("WdF", Wd), ("WuF", Wu)):
            g = par.grad.numpy()
            err = np.linalg.norm(res["grads"][l][key] - g) / np.linalg.norm(g)
            assert err < 1e-10, (l, key, err)
    for d in range(1, cfg.n_layers):
        r = O.step(cfg, layers, head, w["x"], w["labels"], d)
        assert sorted(r["grads"]) == list(range(cfg.n_layers - d, cfg.n_layers))
        for l in r["grads"]:
            for key in ("WdF", "WuF"):
                np.testing.assert_array_equal(r["grads"][l][key], res["grads"][l][key])


def test_fd_tiny_paper_placement():
    cfg = synth.CONFIGS["tiny_paper"]
    _fd_check(cfg, synth.make_workload(cfg, 0), d=1, n_coords=24)
    _fd_check(cfg, _stress_workload(cfg, 3), d=cfg.n_layers, n_coords=12)


def test_encoder_without_adapters_matches_torch_layer_bitwise_identity_invariant():
    """Invariant: zero W_up reproduces the frozen model exactly (Eq. 1 adds 0); the frozen
    model itself matches torch's TransformerEncoderLayer."""
    cfg = _small_enc_cfg()
    w = synth.make_workload(cfg, 1)
    layers, head = O.to_f64_params(w["layers"], w["head"])
    frozen = O.forward(cfg, layers, head, w["x"], w["labels"], 1, adapters=False)
    h = T(w["x"])
    for P in layers:
        h = _torch_encoder_layer(cfg, P, adapters=False)(h)
    np.testing.assert_allclose(frozen["y"], h.reshape(-1, cfg.hidden).detach().numpy(),
                               rtol=1e-11, atol=1e-12)
    for P in layers:
        P["WuA"][:] = 0.0
        P["WuF"][:] = 0.0
    zeroed = O.forward(cfg, layers, head, w["x"], w["labels"], 1, adapters=True)
    np.testing.assert_array_equal(zeroed["y"], frozen["y"])
    np.testing.assert_array_equal(zeroed["logits"], frozen["logits"])
    assert zeroed["loss"] == frozen["loss"]


def test_decoder_zero_up_projection_is_frozen_model():
    cfg = synth.CONFIGS["tiny_dec"]
    w = synth.make_workload(cfg, 2)
    layers, head = O.to_f64_params(w["layers"], w["head"])
    frozen = O.forward(cfg, layers, head, w["x"], w["labels"], 1, adapters=False)
    for P in layers:
        P["WuA"][:] = 0.0
        P["WuF"][:] = 0.0
    zeroed = O.forward(cfg, layers, head, w["x"], w["labels"], 1)
    np.testing.assert_array_equal(zeroed["y"], frozen["y"])
    assert zeroed["loss"] == frozen["loss"]
    r = O.step(cfg, layers, head, w["x"], w["labels"], cfg.n_layers)
    for l in range(cfg.n_layers):
        np.testing.assert_array_equal(r["grads"][l]["WdA"], 0.0)
        np.testing.assert_array_equal(r["grads"][l]["WdF"], 0.0)
        assert np.abs(r["grads"][l]["WuF"]).max() > 0


def test_decoder_branch_wiring_special_cases():
    """Pre-norm residual wiring: with the attention output projection zero, the attention
    branch (and its adapter, which acts on the branch) vanishes and x1 = x exactly; with
    the FFN down projection zero as well, the whole block is the identity."""
    cfg = synth.CONFIGS["tiny_dec"]
    w = _stress_workload(cfg, 3, up_std=0.3)
    layers, head = O.to_f64_params(w["layers"], w["head"])
    P = layers[0]
    cs = O.rope_tables(cfg.seq, cfg.head_dim, cfg.rope_theta)
    x = O.f64(w["x"]).reshape(cfg.tokens, cfg.hidden)
    P["Wo"][:] = 0.0
    y, c = O.decoder_layer_forward(x, P, cfg, cs)
    np.testing.assert_array_equal(c["rms2"][0], x)          # x1 = x
    P["Wd"][:] = 0.0
    y, c = O.decoder_layer_forward(x, P, cfg, cs)
    np.testing.assert_array_equal(y, x)
    # with the down projection alone zero, the block output is x1 (adapter F sees f = 0)
    w2 = _stress_workload(cfg, 3, up_std=0.3)
    P2 = O.to_f64_params(w2["layers"], w2["head"])[0][0]
    P2["Wd"][:] = 0.0
    y, c = O.decoder_layer_forward(x, P2, cfg, cs)
    np.testing.assert_array_equal(y, c["rms2"][0])


# ----------------------------------------------------------------------------------------
# decoder block wiring: closed forms and properties a wrong wiring breaks
# ----------------------------------------------------------------------------------------

def _dec_block(seed=3, up_std=0.3):
    cfg = synth.CONFIGS["tiny_dec"]
    w = _stress_workload(cfg, seed, up_std=up_std)
    P = O.to_f64_params(w["layers"], w["head"])[0][0]
    cs = O.rope_tables(cfg.seq, cfg.head_dim, cfg.rope_theta)
    x = O.f64(w["x"]).reshape(cfg.tokens, cfg.hidden)
    return cfg, P, cs, x


def _dec_out(x, P, cfg, cs):
    # through the module attribute, so that a planted replacement is what runs
    return O.decoder_layer_forward(x, P, cfg, cs)[0]


def test_decoder_norm_gains_zero_close_each_branch():
    """Pre-norm wiring: every projection of a branch reads that branch's RMSNorm output.
    With the first gain zero, q = k = v = 0, so the attention branch and its adapter give
    exactly zero and the block (with the down projection zero too) is the identity; with
    the second gain zero, gate = up = 0 and the block output is x1, the same as with the
    down projection zero."""
    cfg, P, cs, x = _dec_block()
    Q = {k: v.copy() for k, v in P.items()}
    Q["rms1_g"][:] = 0.0
    Q["Wd"][:] = 0.0
    np.testing.assert_array_equal(_dec_out(x, Q, cfg, cs), x)
    Q = {k: v.copy() for k, v in P.items()}
    Q["rms2_g"][:] = 0.0
    R = {k: v.copy() for k, v in P.items()}
    R["Wd"][:] = 0.0
    y_gain0, y_down0 = _dec_out(x, Q, cfg, cs), _dec_out(x, R, cfg, cs)
    np.testing.assert_array_equal(y_gain0, y_down0)
    assert np.abs(y_gain0 - x).max() > 1e-3       # the attention branch is live


def test_decoder_uniform_causal_attention_closed_form():
    """With Wq = Wk = 0 every score is zero, so causal attention averages the values of
    positions 0..t.  With Wo = I, no attention-branch adapter and Wd = 0 the block output
    minus its input is that running mean of RMSNorm(x) Wv^T (torch's rms_norm)."""
    cfg, P, cs, x = _dec_block()
    H, B, S = cfg.hidden, cfg.batch, cfg.seq
    P["Wq"][:] = 0.0
    P["Wk"][:] = 0.0
    P["Wo"][:] = np.eye(H)
    P["WuA"][:] = 0.0
    P["Wd"][:] = 0.0
    n1 = Fnn.rms_norm(T(x), (H,), T(P["rms1_g"]), eps=cfg.norm_eps).numpy()
    v = (n1 @ P["Wv"].T).reshape(B, S, H)
    mean = np.cumsum(v, axis=1) / np.arange(1, S + 1)[None, :, None]
    np.testing.assert_allclose(_dec_out(x, P, cfg, cs) - x, mean.reshape(B * S, H),
                               rtol=1e-10, atol=1e-12)


def test_decoder_block_is_causal():
    """Changing the inputs at positions > t leaves every output at positions <= t
    unchanged (the mask hides the future), while the later outputs do change."""
    cfg, P, cs, x = _dec_block()
    B, S, H = cfg.batch, cfg.seq, cfg.hidden
    y = _dec_out(x, P, cfg, cs).reshape(B, S, H)
    t = S // 3
    x2 = x.reshape(B, S, H).copy()
    x2[:, t + 1:, :] += rng(9).normal(size=x2[:, t + 1:, :].shape)
    y2 = _dec_out(x2.reshape(B * S, H), P, cfg, cs).reshape(B, S, H)
    np.testing.assert_allclose(y2[:, :t + 1], y[:, :t + 1], rtol=1e-12, atol=1e-13)
    assert np.abs(y2[:, t + 1:] - y[:, t + 1:]).max() > 1e-2


def test_decoder_branches_are_scale_invariant():
    """RMSNorm(c x) = RMSNorm(x) for c > 0 (up to eps, 1e-6 against a mean square near 1),
    so a branch whose projections all read its norm output adds the same increment for x
    and for 3x: with Wd = 0 the attention branch, with Wo = 0 the FFN branch."""
    cfg, P, cs, x = _dec_block()
    for zero in ("Wd", "Wo"):
        Q = {k: v.copy() for k, v in P.items()}
        Q[zero][:] = 0.0
        inc1 = _dec_out(x, Q, cfg, cs) - x
        inc3 = _dec_out(3.0 * x, Q, cfg, cs) - 3.0 * x
        assert np.abs(inc1).max() > 1e-3
        np.testing.assert_allclose(inc3, inc1, rtol=1e-5, atol=1e-5 * np.abs(inc1).max())


def test_decoder_heads_are_separable():
    """Multi-head attention: head h's output depends only on head h's rows of Wq, Wk and
    Wv (RoPE rotates pairs inside one head).  With Wo reading head 0 only and Wd = 0,
    redrawing the other heads' projection rows leaves the block output unchanged."""
    cfg, P, cs, x = _dec_block()
    dh = cfg.head_dim
    P["Wo"][:, dh:] = 0.0
    P["Wd"][:] = 0.0
    y = _dec_out(x, P, cfg, cs)
    r = rng(11)
    for key in ("Wq", "Wk", "Wv"):
        P[key][dh:, :] = r.normal(size=P[key][dh:, :].shape) * 0.2
    np.testing.assert_allclose(_dec_out(x, P, cfg, cs), y, rtol=1e-12, atol=1e-13)


# ----------------------------------------------------------------------------------------
# finite differences (brute force) on the tiny configs
# ----------------------------------------------------------------------------------------

def _fd_check(cfg, w, d, n_coords=48, eps=1e-2, tol=1e-6, seed=0, zero_keys=()):
    """Central differences against the oracle's gradients.  ``zero_keys`` name head
    parameters the loss does not depend on (their gradient must be zero both ways)."""
    layers, head = O.to_f64_params(w["layers"], w["head"])
    res = O.step(cfg, layers, head, w["x"], w["labels"], d)
    k = cfg.n_layers - d
    fwd = O.forward(cfg, layers, head, w["x"], w["labels"], cfg.n_layers)
    h_k = fwd["inputs"][k]

    def loss():   # layers below k do not move, so start from the cached input of layer k
        return O.forward(cfg, layers, head, None, w["labels"], d, start_layer=k, h0=h_k)["loss"]

    r = rng(seed)
    targets = [(l, key) for l in range(k, cfg.n_layers) for key in synth.adapter_keys(cfg)]
    if cfg.head_trainable:
        targets += [("head", key) for key in ("Wh", "bh")]
    for l, key in targets:
        par = head[key] if l == "head" else layers[l][key]
        grad = res["head_grads"][key] if l == "head" else res["grads"][l][key]
        n = min(n_coords, par.size)
        idx = r.choice(par.size, n, replace=False)
        fd = np.empty(n)
        for j, i in enumerate(idx):
            th = par.flat[i]
            e = eps * max(1.0, abs(th))
            central = []
            for step in (e, e / 2):
                par.flat[i] = th + step
                lp = loss()
                par.flat[i] = th - step
                lm = loss()
                par.flat[i] = th
                central.append((lp - lm) / (2 * step))
            # Richardson extrapolation of the two central differences: O(e^4) truncation
            fd[j] = (4.0 * central[1] - central[0]) / 3.0
        an = grad.flat[idx]
        if l == "head" and key in zero_keys:
            assert np.abs(an).max() <= 1e-14 and np.abs(fd).max() <= 1e-8, (key, an, fd)
            continue
        err = np.linalg.norm(fd - an) / np.linalg.norm(an)
        assert err <= tol, (l, key, err)
        # per coordinate, against the tensor's scale: a single wrong row or column fails here
        coord = np.abs(fd - an).max() / np.abs(an).max()
        assert coord <= 10 * tol, (l, key, coord)


def test_fd_tiny_encoder_top_layer():
    cfg = synth.CONFIGS["tiny"]
    _fd_check(cfg, synth.make_workload(cfg, 0), d=1)


def test_fd_tiny_encoder_full_depth_stressed():
    cfg = synth.CONFIGS["tiny"]
    _fd_check(cfg, _stress_workload(cfg, 0), d=cfg.n_layers, n_coords=24)


def test_fd_tiny_span_encoder_top_layer_and_full_depth():
    # a common shift of all start (or end) logits of a sequence leaves its softmax
    # unchanged, so the span head's bias gets no gradient at all
    cfg = synth.CONFIGS["tiny_span"]
    _fd_check(cfg, synth.make_workload(cfg, 0), d=1, n_coords=24, zero_keys=("bh",))
    _fd_check(cfg, _stress_workload(cfg, 2), d=cfg.n_layers, n_coords=12, zero_keys=("bh",))


def test_fd_tiny_decoder_top_layer_and_full_depth():
    cfg = synth.CONFIGS["tiny_dec"]
    _fd_check(cfg, synth.make_workload(cfg, 0), d=1, n_coords=24)
    _fd_check(cfg, _stress_workload(cfg, 1, up_std=0.1), d=cfg.n_layers, n_coords=16)


def test_fd_directional_all_adapters():
    """64 random directions over every adapter weight at d = L."""
    for name in ("tiny", "tiny_dec"):
        cfg = synth.CONFIGS[name]
        w = synth.make_workload(cfg, 5)
        layers, head = O.to_f64_params(w["layers"], w["head"])
        res = O.step(cfg, layers, head, w["x"], w["labels"], cfg.n_layers)
        r = rng(9)
        keys = [(l, k) for l in range(cfg.n_layers) for k in synth.ADAPTER_KEYS]
        base = {lk: layers[lk[0]][lk[1]].copy() for lk in keys}
        errs, mags = [], []
        for _ in range(64):
            dirs = {lk: r.normal(size=base[lk].shape) for lk in keys}
            norm = np.sqrt(sum(np.sum(v * v) for v in dirs.values()))
            dirs = {lk: v / norm for lk, v in dirs.items()}
            an = sum(np.sum(res["grads"][l][k] * dirs[(l, k)]) for l, k in keys)
            central = []
            for e in (1e-2, 5e-3):
                vals = []
                for s in (+1, -1):
                    for (l, k) in keys:
                        layers[l][k] = base[(l, k)] + s * e * dirs[(l, k)]
                    vals.append(O.forward(cfg, layers, head, w["x"], w["labels"], 1)["loss"])
                central.append((vals[0] - vals[1]) / (2 * e))
            fd = (4.0 * central[1] - central[0]) / 3.0
            errs.append(fd - an)
            mags.append(an)
        for (l, k) in keys:
            layers[l][k] = base[(l, k)]
        errs, mags = np.array(errs), np.array(mags)
        assert np.linalg.norm(errs) / np.linalg.norm(mags) < 1e-6, name


# ----------------------------------------------------------------------------------------
# the early-stopped backward (Algorithm 1) and its invariants
# ----------------------------------------------------------------------------------------

@pytest.mark.parametrize("name", ["tiny", "tiny_dec", "mid_enc_f32"])
def test_truncated_equals_full_and_nothing_below_k(name):
    """Invariants 2 and 3: for every depth d, gradients of layers >= k equal those of the
    full backward bitwise, and no gradient exists for layers < k or for frozen weights."""
    cfg = synth.CONFIGS[name]
    w = synth.make_workload(cfg, 0)
    layers, head = O.to_f64_params(w["layers"], w["head"])
    full = O.step(cfg, layers, head, w["x"], w["labels"], cfg.n_layers)
    for d in range(1, cfg.n_layers + 1):
        r = O.step(cfg, layers, head, w["x"], w["labels"], d)
        k = cfg.n_layers - d
        assert sorted(r["grads"]) == list(range(k, cfg.n_layers))
        for l in range(k, cfg.n_layers):
            assert sorted(r["grads"][l]) == sorted(synth.ADAPTER_KEYS)
            for key in synth.ADAPTER_KEYS:
                np.testing.assert_array_equal(r["grads"][l][key], full["grads"][l][key])
        assert r["loss"] == full["loss"]
        np.testing.assert_array_equal(r["logits"], full["logits"])
        if cfg.head_trainable:
            for key in r["head_grads"]:
                np.testing.assert_array_equal(r["head_grads"][key], full["head_grads"][key])
        else:
            assert r["head_grads"] == {}


def test_backward_below_saved_depth_is_refused():
    cfg = synth.CONFIGS["tiny"]
    w = synth.make_workload(cfg, 0)
    layers, head = O.to_f64_params(w["layers"], w["head"])
    fwd = O.forward(cfg, layers, head, w["x"], w["labels"], 1)
    with pytest.raises(ValueError):
        O.backward_truncated(cfg, layers, fwd, 0)


def test_paper_ring_example_fig2():
    """Section III-A / Fig. 2: 4:5:2:3 blocks over four clients at depth 3.  The backward of
    the step covers exactly the blocks owned by u4 (the terminator), u2 and u3 do none."""
    ex = json.load(open(os.path.join(GOLDEN, "ring_example.json")))
    L = sum(ex["assignment"])
    owner = []
    for u, n in enumerate(ex["assignment"]):
        owner += ["u%d" % (u + 1)] * n
    cfg = synth.ModelCfg("encoder", L, 16, 2, 32, 4, 2, 2, 4, "f32")
    w = synth.make_workload(cfg, 0)
    layers, head = O.to_f64_params(w["layers"], w["head"])
    r = O.step(cfg, layers, head, w["x"], w["labels"], ex["depth"])
    blocks = sorted(r["grads"])
    assert [b + 1 for b in blocks] == ex["backward_blocks_1based"]
    assert owner[r["k"]] == ex["terminator"]
    with_bwd = sorted({owner[b] for b in blocks})
    assert ["u1"] + with_bwd == ex["backward_clients"]   # u1 is the initiator (loss, head)
    assert sorted(set(owner) - set(with_bwd) - {"u1"}) == ex["clients_without_backward"]


def test_schedule_section4():
    ex = json.load(open(os.path.join(GOLDEN, "schedule_section4.json")))
    for s, d in ex["samples"]:
        assert O.unfreezing_depth(s, ex["interval"], ex["d0"], 24) == d


# ----------------------------------------------------------------------------------------
# Adam
# ----------------------------------------------------------------------------------------

def test_adam_matches_torch_and_late_start():
    r = rng(11)
    p0 = r.normal(size=(6, 5))
    grads = [r.normal(size=(6, 5)) for _ in range(5)]
    pt = torch.nn.Parameter(T(p0))
    opt_t = torch.optim.Adam([pt], lr=1e-4, betas=(0.9, 0.999), eps=1e-8)
    opt = O.Adam(lr=1e-4)
    p = p0.copy()
    for g in grads:
        pt.grad = T(g)
        opt_t.step()
        p = opt.update("w", p, g)
    np.testing.assert_allclose(p, pt.detach().numpy(), rtol=1e-14, atol=1e-16)
    # a parameter first updated later starts at t = 1: its first step is lr * sign-ish(g)
    q = opt.update("late", np.zeros(3), np.array([2.0, -3.0, 0.5]))
    np.testing.assert_allclose(q, -1e-4 * np.array([1.0, -1.0, 1.0]), rtol=1e-6)
    assert opt.state["late"][2] == 1 and opt.state["w"][2] == 5


def test_train_updates_only_unfrozen():
    cfg = synth.CONFIGS["tiny"]
    w = synth.make_workload(cfg, 0)
    layers, head = O.to_f64_params(w["layers"], w["head"])
    before = [{k: v.copy() for k, v in p.items()} for p in layers]
    opt = O.Adam(lr=1e-4)
    O.train(cfg, layers, head, [(w["x"], w["labels"])], [1], opt)
    for key in before[0]:
        np.testing.assert_array_equal(layers[0][key], before[0][key])
    for key in before[1]:
        if key in synth.ADAPTER_KEYS:
            assert not np.array_equal(layers[1][key], before[1][key])
        else:
            np.testing.assert_array_equal(layers[1][key], before[1][key])


# ----------------------------------------------------------------------------------------
# the pins catch plausible mistakes planted in the oracle (CPU only)
# ----------------------------------------------------------------------------------------

def test_planted_mistakes_are_caught(monkeypatch):
    good_adapter_bwd = O.adapter_backward

    def dropped_residual(g, h, z, W_down, W_up, need_dh=True):
        dh, dWd, dWu = good_adapter_bwd(g, h, z, W_down, W_up, need_dh)
        return (dh - g if dh is not None else None), dWd, dWu

    monkeypatch.setattr(O, "adapter_backward", dropped_residual)
    with pytest.raises(AssertionError):
        test_encoder_stack_matches_torch_layers_with_autograd()
    monkeypatch.setattr(O, "adapter_backward", good_adapter_bwd)

    good_rope_bwd = O.rope_backward
    monkeypatch.setattr(O, "rope_backward", lambda dt, c, s: good_rope_bwd(dt, c, -s))
    with pytest.raises(AssertionError):
        cfg = synth.CONFIGS["tiny_dec"]
        _fd_check(cfg, _stress_workload(cfg, 1, up_std=0.1), d=cfg.n_layers, n_coords=4)
    monkeypatch.setattr(O, "rope_backward", good_rope_bwd)

    good_attn_bwd = O.attention_backward

    def transposed(dO, q, k, v, p):
        dq, dk, dv = good_attn_bwd(dO, q, k, v, p)
        return dq, dk, p @ dO          # P instead of P^T
    monkeypatch.setattr(O, "attention_backward", transposed)
    with pytest.raises(AssertionError):
        test_attention_matches_sdpa(False)
    monkeypatch.setattr(O, "attention_backward", good_attn_bwd)

    good_ln = O.layer_norm

    def unbiased_var(s, gamma, beta, eps):
        _, (xhat, rstd) = good_ln(s, gamma, beta, eps)
        c = np.sqrt((s.shape[-1] - 1.0) / s.shape[-1])
        return xhat * c * gamma + beta, (xhat * c, rstd * c)
    monkeypatch.setattr(O, "layer_norm", unbiased_var)
    with pytest.raises(AssertionError):
        test_encoder_without_adapters_matches_torch_layer_bitwise_identity_invariant()

    # span head: start and end labels swapped, or the two cross-entropies summed instead of
    # averaged; the torch comparison and the finite differences must both notice
    good_span = O.encoder_span_head
    monkeypatch.setattr(O, "encoder_span_head",
                        lambda y, head, labels, cfg: good_span(y, head, np.asarray(labels)[:, ::-1], cfg))
    with pytest.raises(AssertionError):
        test_span_head_matches_torch_autograd()

    def summed(y, head, labels, cfg):
        loss, logits, dy, g = good_span(y, head, labels, cfg)
        return 2 * loss, logits, dy, g
    monkeypatch.setattr(O, "encoder_span_head", summed)
    with pytest.raises(AssertionError):
        test_span_head_matches_torch_autograd()
    with pytest.raises(AssertionError):
        cfg = synth.CONFIGS["tiny_span"]
        _fd_check(cfg, synth.make_workload(cfg, 0), d=1, n_coords=4, zero_keys=("bh",))
    monkeypatch.setattr(O, "encoder_span_head", good_span)

    # decoder block wiring: q or v projected from x instead of RMSNorm(x), gate/up fed by
    # x1 instead of RMSNorm(x1), the causal mask reversed, RoPE applied across the merged
    # heads; each fails one of the wiring pins
    good_dec = O.decoder_layer_forward
    x_case = _dec_block()
    np.testing.assert_array_equal(_decoder_variant(None)(*_dec_args(x_case))[0],
                                  good_dec(*_dec_args(x_case))[0])
    wiring_pins = (test_decoder_norm_gains_zero_close_each_branch,
                   test_decoder_uniform_causal_attention_closed_form,
                   test_decoder_block_is_causal,
                   test_decoder_branches_are_scale_invariant,
                   test_decoder_heads_are_separable)
    for mistake in ("q_from_x", "v_from_x", "gate_up_from_x1", "mask_reversed", "rope_merged"):
        monkeypatch.setattr(O, "decoder_layer_forward", _decoder_variant(mistake))
        failed = 0
        for pin in wiring_pins:
            try:
                pin()
            except AssertionError:
                failed += 1
        assert failed >= 1, mistake
        monkeypatch.setattr(O, "decoder_layer_forward", good_dec)


def _dec_args(case):
    cfg, P, cs, x = case
    return x, P, cfg, cs


def _decoder_variant(mistake):
    """The oracle's decoder block forward restated with one wiring mistake planted (None:
    no mistake, which must equal the oracle bitwise)."""
    def fwd(x, P, cfg, rope_cs, adapters=True):
        B, S, nh, H = cfg.batch, cfg.seq, cfg.n_heads, cfg.hidden
        cos, sin = rope_cs
        n1, rms1 = O.rms_norm(x, P["rms1_g"], cfg.norm_eps)
        qin = x if mistake == "q_from_x" else n1
        vin = x if mistake == "v_from_x" else n1
        if mistake == "rope_merged":
            # rotate-half pairs (i, i + H/2) across the whole row, before the head split
            ang_q = O.rope(np.stack([qin @ P["Wq"].T]), *O.rope_tables(B * S, H, cfg.rope_theta))[0]
            ang_k = O.rope(np.stack([n1 @ P["Wk"].T]), *O.rope_tables(B * S, H, cfg.rope_theta))[0]
            q = O.split_heads(ang_q, B, S, nh)
            k = O.split_heads(ang_k, B, S, nh)
        else:
            q = O.rope(O.split_heads(qin @ P["Wq"].T, B, S, nh), cos, sin)
            k = O.rope(O.split_heads(n1 @ P["Wk"].T, B, S, nh), cos, sin)
        v = O.split_heads(vin @ P["Wv"].T, B, S, nh)
        if mistake == "mask_reversed":
            Of, p = O.attention(q[:, :, ::-1], k[:, :, ::-1], v[:, :, ::-1], causal=True)
            Oo, p = Of[:, :, ::-1], p[:, :, ::-1, ::-1]
        else:
            Oo, p = O.attention(q, k, v, causal=True)
        a = O.merge_heads(Oo) @ P["Wo"].T
        a2, zA = O.adapter_forward(a, P["WdA"], P["WuA"]) if adapters else (a, None)
        x1 = x + a2
        n2, rms2 = O.rms_norm(x1, P["rms2_g"], cfg.norm_eps)
        fin = x1 if mistake == "gate_up_from_x1" else n2
        gate = fin @ P["Wg"].T
        up = fin @ P["Wu"].T
        f = (O.silu(gate) * up) @ P["Wd"].T
        f2, zF = O.adapter_forward(f, P["WdF"], P["WuF"]) if adapters else (f, None)
        cache = dict(rms1=rms1, q=q, k=k, v=v, p=p, a=a, zA=zA, rms2=rms2, gate=gate, up=up,
                     f=f, zF=zF)
        return x1 + f2, cache
    return fwd
