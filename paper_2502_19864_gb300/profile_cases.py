"""Small, self-contained launch cases for profiler captures (ncu) of single kernels.

  python -m paper_2502_19864_gb300.profile_cases gemm M N K [--reps R] [--gelu] [--epi E]
      R launches of the tensor-core GEMM C[M,N] = A[M,K] B[N,K]^T (bf16, via ra_gemm_bf16);
      --gelu adds the bias + GELU epilogue (writes C and GELU(C)); --epi selects one of the
      step's epilogues through ra_gemm_bf16_epi: gelu_g (GELU and GELU'), mul (times a bf16
      operand), f32 (fp32 output)
  python -m paper_2502_19864_gb300.profile_cases step CONFIG D [--reps R] [--layers N]
      R eager steps (forward, early-stopped backward, update) of a synthetic workload; with
      --layers, the workload's per-layer shapes on N layers (a smaller device footprint)

Inputs are seeded synthetic data; every call goes through the C ABI.
"""
from __future__ import annotations

import argparse
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))


def gemm_epi_case(M, N, K, reps, epi):
    import torch
    from paper_2502_19864_gb300 import ringada as R
    g = torch.Generator().manual_seed(0)
    A = torch.randn(M, K, generator=g).to(torch.bfloat16).cuda()
    B = (torch.randn(N, K, generator=g) * 0.05).to(torch.bfloat16).cuda()
    bias = torch.randn(N, generator=g).float().cuda()
    aux = torch.rand(M, N, generator=g).to(torch.bfloat16).cuda()
    f32 = epi == "f32"
    C = torch.empty(M, N, dtype=torch.float32 if f32 else torch.bfloat16, device="cuda")
    C2 = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    kind = {"gelu_g": R.RA_EPI_BIAS_GELU_G, "mul": R.RA_EPI_MUL, "f32": R.RA_EPI_STORE}[epi]
    for _ in range(reps):
        R.ra_gemm_bf16_epi(A.data_ptr(), B.data_ptr(), M, N, K, kind,
                           bias.data_ptr() if epi == "gelu_g" else None,
                           aux.data_ptr() if epi == "mul" else None, C.data_ptr(),
                           R.RA_F32 if f32 else R.RA_BF16, C2.data_ptr() if epi == "gelu_g" else None)
    torch.cuda.synchronize()
    print("gemm %s %dx%dx%d x%d done" % (epi, M, N, K, reps))


def gemm_case(M, N, K, reps, gelu=False):
    import torch
    from paper_2502_19864_gb300 import ringada as R
    g = torch.Generator().manual_seed(0)
    A = torch.randn(M, K, generator=g).to(torch.bfloat16).cuda()
    B = (torch.randn(N, K, generator=g) * 0.05).to(torch.bfloat16).cuda()
    C = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    bias = torch.randn(N, generator=g).float().cuda() if gelu else None
    G = torch.empty(M, N, dtype=torch.bfloat16, device="cuda") if gelu else None
    for _ in range(reps):
        R.ra_gemm_bf16(A.data_ptr(), B.data_ptr(), C.data_ptr(), M, N, K,
                       bias.data_ptr() if gelu else None, G.data_ptr() if gelu else None)
    torch.cuda.synchronize()
    print("gemm %dx%dx%d x%d done" % (M, N, K, reps))


def step_case(name, d, reps, layers=None):
    import dataclasses
    import torch
    import synth
    from paper_2502_19864_gb300 import ringada as R
    cfg = synth.CONFIGS[name]
    if layers:
        cfg = dataclasses.replace(cfg, n_layers=layers)
    w = synth.make_workload(cfg, 0)
    if cfg.arch == "decoder":
        arch = R.RA_DECODER_PRENORM
    else:
        arch = R.RA_ENCODER_POSTLN_SPAN if cfg.head == "span" else R.RA_ENCODER_POSTLN
    placement = R.RA_ADAPTERS_POST_FFN if cfg.adapters == "paper" else R.RA_ADAPTERS_HOULSBY
    m = R.Model(R.make_cfg(arch, cfg.n_layers, cfg.hidden, cfg.n_heads, cfg.ffn, cfg.n_out,
                           cfg.batch, cfg.seq, R.RA_BF16 if cfg.dtype == "bf16" else R.RA_F32,
                           int(cfg.head_trainable), 0, cfg.norm_eps, cfg.rope_theta, placement),
                cfg.adapter_dim)
    m.set_weights(w["layers"], w["head"])
    dt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    x = torch.tensor(w["x"], dtype=torch.float32).to(dt).cuda()
    labels = torch.tensor(w["labels"], dtype=torch.int32).cuda()
    loss = torch.zeros(1, dtype=torch.float32, device="cuda")
    R.ra_set_unfrozen_depth(m.ctx, d)
    for _ in range(reps):
        R.ra_forward(m.ctx, x.data_ptr(), labels.data_ptr(), cfg.batch, cfg.seq, loss.data_ptr())
        R.ra_backward_truncated(m.ctx, cfg.n_layers - d)
        R.ra_adapter_update(m.ctx)
    R.ra_sync_status(m.ctx)
    print("step %s d=%d x%d loss %.6f" % (name, d, reps, loss.item()))
    m.close()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("case", choices=["gemm", "step"])
    ap.add_argument("args", nargs="+")
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--gelu", action="store_true")
    ap.add_argument("--layers", type=int, default=None)
    ap.add_argument("--epi", default=None, choices=["gelu_g", "mul", "f32"])
    a = ap.parse_args()
    import __graft_entry__
    __graft_entry__.build()
    if a.case == "gemm":
        M, N, K = (int(v) for v in a.args[:3])
        if a.epi:
            gemm_epi_case(M, N, K, a.reps, a.epi)
        else:
            gemm_case(M, N, K, a.reps, a.gelu)
    else:
        step_case(a.args[0], int(a.args[1]), a.reps, a.layers)


if __name__ == "__main__":
    main()
