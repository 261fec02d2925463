"""Shared helpers of the GPU tests: run the CUDA path through the C ABI on a synthetic
workload and compare it with the fp64 oracle."""
import numpy as np

import synth
from oracle import ringada_oracle as O
from paper_2502_19864_gb300 import ringada as R

# tolerances of the parity bar
F32_TOL = 1e-4          # max |gpu - oracle| / max |oracle|, per tensor (fp32 models)
# element-wise relative error of fp32 models, max_i |gpu_i - oracle_i| / max(|oracle_i|,
# floor): relative error is undefined at zeros, so elements below the floor (a stated
# fraction of the tensor's largest magnitude) are measured against the floor instead
F32_ELEM_FLOOR = 1e-2   # floor = F32_ELEM_FLOOR * max |oracle|
F32_ELEM_TOL = 1e-3
BF16_LOSS_TOL = 2e-2    # relative, loss; normwise, logits (bf16 models)
BF16_GRAD_TOL = 5e-2    # normwise, per adapter/head gradient tensor (bf16 models)


def ra_arch(cfg):
    if cfg.arch == "decoder":
        return R.RA_DECODER_PRENORM
    return R.RA_ENCODER_POSTLN_SPAN if cfg.head == "span" else R.RA_ENCODER_POSTLN


def ra_cfg(cfg, max_depth=0, max_batch=None, max_seq=None):
    arch = ra_arch(cfg)
    dt = R.RA_BF16 if cfg.dtype == "bf16" else R.RA_F32
    placement = R.RA_ADAPTERS_POST_FFN if cfg.adapters == "paper" else R.RA_ADAPTERS_HOULSBY
    return R.make_cfg(arch, cfg.n_layers, cfg.hidden, cfg.n_heads, cfg.ffn, cfg.n_out,
                      max_batch or cfg.batch, max_seq or cfg.seq, dt, int(cfg.head_trainable),
                      max_depth, cfg.norm_eps, cfg.rope_theta, placement)


class GpuStepper:
    """One context on cuda:0 loaded with a synthetic workload."""

    def __init__(self, cfg, w, max_depth=0, want_logits=True, max_batch=None, max_seq=None):
        import torch
        self.torch = torch
        self.cfg = cfg
        self.w = w
        self.model = R.Model(ra_cfg(cfg, max_depth, max_batch, max_seq), cfg.adapter_dim,
                             device="cuda:0")
        self.model.set_weights(w["layers"], w["head"])
        dt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
        self.x = torch.tensor(w["x"], dtype=torch.float32).to(dt).cuda()
        self.labels = torch.tensor(w["labels"], dtype=torch.int32).cuda()
        self.loss = torch.zeros(1, dtype=torch.float32, device="cuda")
        rows = cfg.batch if (cfg.arch == "encoder" and cfg.head == "cls") else cfg.tokens
        self.logits = torch.zeros(rows, cfg.n_out, dtype=torch.float32, device="cuda") if want_logits else None

    @property
    def ctx(self):
        return self.model.ctx

    def set_batch(self, x, labels):
        self.x.copy_(self.torch.tensor(x).to(self.x.dtype))
        self.labels.copy_(self.torch.tensor(labels))

    def forward(self, d):
        R.ra_set_unfrozen_depth(self.ctx, d)
        R.ra_forward(self.ctx, self.x.data_ptr(), self.labels.data_ptr(), self.cfg.batch,
                     self.cfg.seq, self.loss.data_ptr(),
                     self.logits.data_ptr() if self.logits is not None else None)

    def step(self, d, update=False):
        self.forward(d)
        R.ra_backward_truncated(self.ctx, self.cfg.n_layers - d)
        if update:
            R.ra_adapter_update(self.ctx)
        R.ra_sync_status(self.ctx)
        return self.loss.item()

    def grads(self, k):
        out = {}
        for l in range(k, self.cfg.n_layers):
            out[l] = {key: self.model.grad(l, key).double().cpu().numpy().reshape(
                synth.param_shape(self.cfg, key)) for key in synth.adapter_keys(self.cfg)}
        return out

    def head_grads(self):
        if not self.cfg.head_trainable:
            return {}
        return {key: self.model.grad(-1, key).double().cpu().numpy().reshape(
            synth.param_shape(self.cfg, key)) for key in ("Wh", "bh")}

    def close(self):
        self.model.close()


def oracle_full(cfg, w):
    """Oracle forward at full depth plus the full backward (every layer's gradients)."""
    layers, head = O.to_f64_params(w["layers"], w["head"])
    return O.step(cfg, layers, head, w["x"], w["labels"], cfg.n_layers)


def rel_max(a, b):
    return float(np.abs(a - b).max() / max(np.abs(b).max(), 1e-30))


def rel_elem(a, b, floor_frac=F32_ELEM_FLOOR):
    floor = floor_frac * max(float(np.abs(b).max()), 1e-30)
    return float((np.abs(a - b) / np.maximum(np.abs(b), floor)).max())


def rel_norm(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


# The span head's bias gets no gradient (a common shift of a sequence's start or end logits
# leaves its softmax unchanged): the GPU's fp32 sum of dlogits must be zero up to rounding.
SPAN_BIAS_GRAD_ABS = 1e-5


def check_step(cfg, gpu_loss, gpu_logits, gpu_grads, gpu_head, ref, k):
    """Asserts the parity bar; returns the worst errors for reporting."""
    report = {}
    if getattr(cfg, "head", "cls") == "span" and "bh" in gpu_head:
        gpu_head = dict(gpu_head)
        report["head_bh_abs"] = float(np.abs(gpu_head.pop("bh")).max())
        assert report["head_bh_abs"] <= SPAN_BIAS_GRAD_ABS, report
        assert np.abs(ref["head_grads"]["bh"]).max() <= 1e-14
    if cfg.dtype == "f32":
        report["loss"] = abs(gpu_loss - ref["loss"]) / abs(ref["loss"])
        assert report["loss"] <= F32_TOL, report
        if gpu_logits is not None:
            report["logits"] = rel_max(gpu_logits, ref["logits"])
            assert report["logits"] <= F32_TOL, report
            report["logits_elem"] = rel_elem(gpu_logits, ref["logits"])
            assert report["logits_elem"] <= F32_ELEM_TOL, report
        for l in range(k, cfg.n_layers):
            for key in synth.adapter_keys(cfg):
                e = rel_max(gpu_grads[l][key], ref["grads"][l][key])
                report["g%d%s" % (l, key)] = e
                assert e <= F32_TOL, (l, key, e)
                e = rel_elem(gpu_grads[l][key], ref["grads"][l][key])
                report["g%d%s_elem" % (l, key)] = e
                assert e <= F32_ELEM_TOL, (l, key, "elementwise", e)
        for key, g in gpu_head.items():
            e = rel_max(g, ref["head_grads"][key])
            report["head" + key] = e
            assert e <= F32_TOL, (key, e)
            e = rel_elem(g, ref["head_grads"][key])
            report["head%s_elem" % key] = e
            assert e <= F32_ELEM_TOL, (key, "elementwise", e)
    else:
        report["loss"] = abs(gpu_loss - ref["loss"]) / abs(ref["loss"])
        assert report["loss"] <= BF16_LOSS_TOL, report
        if gpu_logits is not None:
            report["logits"] = rel_norm(gpu_logits, ref["logits"])
            assert report["logits"] <= BF16_LOSS_TOL, report
        for l in range(k, cfg.n_layers):
            for key in synth.adapter_keys(cfg):
                e = rel_norm(gpu_grads[l][key], ref["grads"][l][key])
                report["g%d%s" % (l, key)] = e
                assert e <= BF16_GRAD_TOL, (l, key, e)
        for key, g in gpu_head.items():
            e = rel_norm(g, ref["head_grads"][key])
            report["head" + key] = e
            assert e <= BF16_GRAD_TOL, (key, e)
    return report
