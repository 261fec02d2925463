"""Edge cases of the step on the GPU (through the C ABI) against the fp64 oracle: one-token
batches (a one-key softmax, single-row tiles everywhere), batches smaller than the context's
capacity, heads with more than two classes, and the exact zero of dW_down when every
up-projection is zero (Eq. 1 differentiated: dz = (g W_up^T) * GELU'(z) = 0)."""
import dataclasses

import numpy as np
import pytest

import synth
from gpu_helpers import GpuStepper, check_step, oracle_full

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


def _parity(cfg, w, depths, **kw):
    ref = oracle_full(cfg, w)
    run = GpuStepper(cfg, w, **kw)
    try:
        for d in depths:
            k = cfg.n_layers - d
            loss = run.step(d)
            logits = run.logits.double().cpu().numpy()
            check_step(cfg, loss, logits, run.grads(k), run.head_grads(), ref, k)
    finally:
        run.close()


@pytest.mark.parametrize("name", ["tiny", "small_enc_bf16", "small_dec_bf16"])
def test_one_token_batch(name):
    cfg = dataclasses.replace(synth.CONFIGS[name], batch=1, seq=1)
    _parity(cfg, synth.make_workload(cfg, 5), [1, cfg.n_layers])


@pytest.mark.parametrize("name,batch,seq", [("small_enc_bf16", 2, 61), ("small_dec_bf16", 1, 117),
                                            ("mid_enc_f32", 2, 30)])
def test_batch_smaller_than_capacity(name, batch, seq):
    big = synth.CONFIGS[name]
    cfg = dataclasses.replace(big, batch=batch, seq=seq)
    _parity(cfg, synth.make_workload(cfg, 6), [1, cfg.n_layers], max_batch=big.batch, max_seq=big.seq)


@pytest.mark.parametrize("classes", [5, 20])
def test_heads_with_more_classes(classes):
    cfg = dataclasses.replace(synth.CONFIGS["tiny"], n_out=classes)
    _parity(cfg, synth.make_workload(cfg, 7), [1, cfg.n_layers])


@pytest.mark.parametrize("name", ["tiny", "small_enc_bf16", "small_dec_bf16"])
def test_zero_up_projection_gives_exactly_zero_down_gradient(name):
    cfg = synth.CONFIGS[name]
    w = synth.make_workload(cfg, 8)
    for p in w["layers"]:
        p["WuA"] = np.zeros_like(p["WuA"])
        p["WuF"] = np.zeros_like(p["WuF"])
    ref = oracle_full(cfg, w)
    run = GpuStepper(cfg, w)
    try:
        loss = run.step(cfg.n_layers)
        grads = run.grads(0)
        check_step(cfg, loss, run.logits.double().cpu().numpy(), grads, run.head_grads(), ref, 0)
        for l in range(cfg.n_layers):
            assert not np.any(grads[l]["WdA"]) and not np.any(grads[l]["WdF"]), l
            assert np.any(grads[l]["WuA"]) and np.any(grads[l]["WuF"]), l
    finally:
        run.close()
