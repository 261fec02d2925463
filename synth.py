"""Seeded synthetic workloads for the adapter fine-tuning step.

This module holds model shapes, random draws in a fixed order and rounding to the storage
type, and nothing of the method's arithmetic.  The CUDA path (through the package binding),
the tests, the bench and the fp64 oracle all take their inputs from here; the oracle never
imports it itself (callers pass it arrays).

Workload recipe (stands in for mBERT on SQuAD, Section IV, which is not available offline):
  * x ~ N(0, 1) hidden states [B, S, H] (no embedding layer; Emb is outside the path),
  * frozen linear weights and biases ~ N(0, 0.02); LayerNorm gamma ~ 1 + N(0, 0.02),
    beta ~ N(0, 0.02); RMSNorm gamma ~ 1 + N(0, 0.02),
  * adapter down-projection ~ N(0, 0.02), up-projection ~ N(0, 1e-3) (Eq. 1 shapes
    W_down [H, m], W_up [m, H]),
  * encoder: 2-class CLS head ~ N(0, 0.02), labels uniform in [0, 2); or a span head
    (start and end logits at every token) ~ N(0, 0.02) with start and end positions drawn
    independently and uniformly in [0, S);
    decoder: frozen vocabulary head, token labels uniform in [0, V),
  * one torch CPU generator, seed 0 unless stated, draws in the order of ``layer_keys``,
    then the head, then x, then the labels; every value is rounded once to the storage
    dtype (round-to-nearest-even for bf16) and kept as float32 holding that exact value.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class ModelCfg:
    arch: str            # "encoder" (post-LN, GELU FFN, CLS head) | "decoder" (pre-RMSNorm, RoPE, SwiGLU)
    n_layers: int
    hidden: int
    n_heads: int
    ffn: int
    adapter_dim: int
    n_out: int           # classes (encoder) or vocabulary (decoder)
    batch: int
    seq: int
    dtype: str           # "f32" | "bf16"
    head_trainable: bool = True
    norm_eps: float = 1e-12
    rope_theta: float = 10000.0
    head: str = "cls"    # encoder head: "cls" (position 0, n_out classes) | "span" (start/end
                         # logits at every position, n_out = 2)
    adapters: str = "houlsby"  # encoder: "houlsby" (attention- and FFN-branch adapters) |
                               # "paper" (one adapter after the FFN add & LayerNorm, Fig. 1)

    @property
    def head_dim(self) -> int:
        return self.hidden // self.n_heads

    @property
    def tokens(self) -> int:
        return self.batch * self.seq


def _enc(L, H, h, F, m, B, S, dtype, C=2):
    return ModelCfg("encoder", L, H, h, F, m, C, B, S, dtype, True, 1e-12)


def _span(L, H, h, F, m, B, S, dtype):
    return ModelCfg("encoder", L, H, h, F, m, 2, B, S, dtype, True, 1e-12, head="span")


def _paper(L, H, h, F, m, B, S, dtype):
    return ModelCfg("encoder", L, H, h, F, m, 2, B, S, dtype, True, 1e-12, adapters="paper")


def _dec(L, H, h, F, m, V, B, S, dtype):
    return ModelCfg("decoder", L, H, h, F, m, V, B, S, dtype, False, 1e-6)


CONFIGS: Dict[str, ModelCfg] = {
    # the five workloads
    "tiny": _enc(2, 128, 2, 512, 16, 4, 32, "f32"),
    "base": _enc(12, 768, 12, 3072, 64, 32, 128, "bf16"),
    "large": _enc(24, 1024, 16, 4096, 64, 32, 256, "bf16"),
    "llama": _dec(16, 2048, 16, 5632, 128, 32000, 8, 1024, "bf16"),
    # small parity cases: several tiles plus ragged tails
    "tiny_dec": _dec(2, 128, 2, 320, 16, 101, 2, 48, "f32"),
    "small_enc_bf16": _enc(3, 256, 4, 1024, 32, 3, 100, "bf16"),
    "small_dec_bf16": _dec(3, 256, 2, 704, 32, 1000, 2, 200, "bf16"),
    "mid_enc_f32": _enc(3, 192, 3, 768, 24, 5, 77, "f32"),
    # span (start/end) head over every token, the shape of extractive question answering
    "tiny_span": _span(2, 128, 2, 512, 16, 4, 32, "f32"),
    "small_span_bf16": _span(3, 256, 4, 1024, 32, 3, 100, "bf16"),
    # the paper's placement: one adapter per block, after the FFN add & LayerNorm
    "tiny_paper": _paper(2, 128, 2, 512, 16, 4, 32, "f32"),
    "small_paper_bf16": _paper(3, 256, 4, 1024, 32, 3, 100, "bf16"),
    # two 128-row key/query blocks with a ragged second block (S = 250)
    "small_enc_s250_bf16": _enc(2, 256, 4, 1024, 32, 2, 250, "bf16"),
    # m = 64 and H = 512: the fused tcgen05 adapter forward over clusters of two CTAs, with a
    # ragged last 128-row tile (T = 300), in both placements
    "small_enc_m64_bf16": _enc(2, 512, 8, 1024, 64, 3, 100, "bf16"),
    "small_paper_m64_bf16": _paper(2, 512, 8, 1024, 64, 3, 100, "bf16"),
    # the BERT-large layer shapes on 2 layers: its FFN-down and dX GEMMs run stream-K, on two
    # streams at once when the next batch's prefix overlaps
    "large_2l": _enc(2, 1024, 16, 4096, 64, 32, 256, "bf16"),
    # the bench workloads' shapes with the other heads / placement (per-kernel profiles)
    "base_span": _span(12, 768, 12, 3072, 64, 32, 128, "bf16"),
    "large_paper": _paper(24, 1024, 16, 4096, 64, 32, 256, "bf16"),
}


ENCODER_LAYER_KEYS = ["Wqkv", "bqkv", "Wo", "bo", "WdA", "WuA", "ln1_g", "ln1_b",
                      "W1", "b1", "W2", "b2", "WdF", "WuF", "ln2_g", "ln2_b"]
DECODER_LAYER_KEYS = ["Wq", "Wk", "Wv", "Wo", "WdA", "WuA", "rms1_g",
                      "Wg", "Wu", "Wd", "WdF", "WuF", "rms2_g"]
ADAPTER_KEYS = ["WdA", "WuA", "WdF", "WuF"]


def layer_keys(cfg: ModelCfg) -> List[str]:
    if cfg.arch == "encoder" and cfg.adapters == "paper":
        return [k for k in ENCODER_LAYER_KEYS if k not in ("WdA", "WuA")]
    return ENCODER_LAYER_KEYS if cfg.arch == "encoder" else DECODER_LAYER_KEYS


def adapter_keys(cfg: ModelCfg) -> List[str]:
    """The trainable adapter matrices of one block."""
    return ["WdF", "WuF"] if cfg.arch == "encoder" and cfg.adapters == "paper" else ADAPTER_KEYS


def head_keys(cfg: ModelCfg) -> List[str]:
    return ["Wh", "bh"] if cfg.arch == "encoder" else ["rmsf_g", "Wh"]


def param_shape(cfg: ModelCfg, key: str):
    H, F, m = cfg.hidden, cfg.ffn, cfg.adapter_dim
    table = {
        "Wqkv": (3 * H, H), "bqkv": (3 * H,), "Wo": (H, H), "bo": (H,),
        "WdA": (H, m), "WuA": (m, H), "WdF": (H, m), "WuF": (m, H),
        "ln1_g": (H,), "ln1_b": (H,), "ln2_g": (H,), "ln2_b": (H,),
        "W1": (F, H), "b1": (F,), "W2": (H, F), "b2": (H,),
        "Wq": (H, H), "Wk": (H, H), "Wv": (H, H),
        "rms1_g": (H,), "rms2_g": (H,), "rmsf_g": (H,),
        "Wg": (F, H), "Wu": (F, H), "Wd": (H, F),
        "Wh": (cfg.n_out, H), "bh": (cfg.n_out,),
    }
    return table[key]


def _draw(gen, key: str, shape):
    if key in ("WuA", "WuF"):
        return torch.randn(shape, generator=gen) * 1e-3
    if key.endswith("_g"):
        return 1.0 + torch.randn(shape, generator=gen) * 0.02
    return torch.randn(shape, generator=gen) * 0.02


def round_to(arr: torch.Tensor, dtype: str) -> np.ndarray:
    """Round once to the storage type; return float32 holding the exact stored value."""
    if dtype == "bf16":
        arr = arr.to(torch.bfloat16).to(torch.float32)
    return arr.to(torch.float32).numpy().copy()


def make_workload(cfg: ModelCfg, seed: int = 0):
    """Weights, inputs and labels for one step, in the fixed draw order.

    Returns dict(layers=[{key: f32 array}], head={key: f32 array}, x=[B,S,H] f32,
    labels=int32 [B] (encoder) or [B,S] (decoder)).
    """
    gen = torch.Generator().manual_seed(seed)
    layers = []
    for _ in range(cfg.n_layers):
        p = {}
        for key in layer_keys(cfg):
            p[key] = round_to(_draw(gen, key, param_shape(cfg, key)), cfg.dtype)
        layers.append(p)
    head = {}
    for key in head_keys(cfg):
        head[key] = round_to(_draw(gen, key, param_shape(cfg, key)), cfg.dtype)
    x = round_to(torch.randn((cfg.batch, cfg.seq, cfg.hidden), generator=gen), cfg.dtype)
    if cfg.arch == "encoder" and cfg.head == "span":
        labels = torch.randint(0, cfg.seq, (cfg.batch, 2), generator=gen)
    elif cfg.arch == "encoder":
        labels = torch.randint(0, cfg.n_out, (cfg.batch,), generator=gen)
    else:
        labels = torch.randint(0, cfg.n_out, (cfg.batch, cfg.seq), generator=gen)
    return dict(layers=layers, head=head, x=x, labels=labels.to(torch.int32).numpy())


def make_batch(cfg: ModelCfg, seed: int):
    """A fresh (x, labels) batch from its own generator, for multi-step runs."""
    gen = torch.Generator().manual_seed(seed)
    x = round_to(torch.randn((cfg.batch, cfg.seq, cfg.hidden), generator=gen), cfg.dtype)
    if cfg.arch == "encoder" and cfg.head == "span":
        labels = torch.randint(0, cfg.seq, (cfg.batch, 2), generator=gen)
    else:
        shape = (cfg.batch,) if cfg.arch == "encoder" else (cfg.batch, cfg.seq)
        labels = torch.randint(0, cfg.n_out, shape, generator=gen)
    labels = labels.to(torch.int32).numpy()
    return x, labels

