"""The next-batch prefix (ra_forward_prefix / ra_forward_suffix): the forward split at the
lowest unfrozen layer k, with the frozen blocks below k on their own scratch buffers
(Section III-A: the forward below the unfreezing depth is independent of the training
above it and can run at the same time; Section III-B.2).

Checked through the C ABI: the split forward gives bitwise the loss, logits and adapter
gradients of ra_forward; the prefix of batch s + 1 run on a second stream while batch s
is in its backward and update gives bitwise the same trajectory as the sequential steps;
and the split calls reject out-of-order use."""
import numpy as np
import pytest

import synth
from paper_2502_19864_gb300 import ringada as R
from gpu_helpers import GpuStepper, ra_cfg

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


class PrefixRun(GpuStepper):
    """A GpuStepper whose context reserves the prefix buffers."""

    def __init__(self, cfg, w):
        import torch
        orig = R.make_cfg

        def with_prefix(*a, **kw):
            kw["prefix_buffers"] = 1
            return orig(*a, **kw)
        R.make_cfg = with_prefix
        try:
            super().__init__(cfg, w)
        finally:
            R.make_cfg = orig
        self.torch = torch

    def split_step(self, d, buf=0, update=False):
        R.ra_set_unfrozen_depth(self.ctx, d)
        R.ra_forward_prefix(self.ctx, self.x.data_ptr(), self.cfg.batch, self.cfg.seq, buf)
        R.ra_forward_suffix(self.ctx, buf, self.labels.data_ptr(), self.loss.data_ptr(),
                            self.logits.data_ptr())
        R.ra_backward_truncated(self.ctx, self.cfg.n_layers - d)
        if update:
            R.ra_adapter_update(self.ctx)
        R.ra_sync_status(self.ctx)
        return self.loss.item()


@pytest.mark.parametrize("name", ["tiny", "small_enc_bf16", "small_paper_bf16", "small_span_bf16"])
def test_split_forward_is_bitwise_the_forward(name):
    cfg = synth.CONFIGS[name]
    run = PrefixRun(cfg, synth.make_workload(cfg, 1))
    try:
        for d in range(1, cfg.n_layers + 1):
            k = cfg.n_layers - d
            l1 = run.step(d)
            lg1 = run.logits.clone()
            g1 = run.grads(k)
            for buf in (0, 1):
                l2 = run.split_step(d, buf)
                assert l2 == l1, (d, buf)
                assert bool((run.logits == lg1).all())
                g2 = run.grads(k)
                for l in g1:
                    for key in g1[l]:
                        np.testing.assert_array_equal(g2[l][key], g1[l][key])
    finally:
        run.close()


@pytest.mark.parametrize("name", ["small_enc_bf16", "large_2l"])
def test_prefix_on_a_second_stream_overlapping_the_backward_matches_sequential_steps(name):
    """Four Adam steps on distinct batches with the unfreezing depth growing from 1 to 2:
    the prefix of batch s + 1 is enqueued on stream B while batch s's suffix, backward and
    update run on stream A (events order the shared buffers), against the same steps run
    one after the other through ra_forward.  With the BERT-large layer shapes the stream-K
    GEMMs of both streams run at the same time, each on its own scratch."""
    import torch
    cfg = synth.CONFIGS[name]
    w = synth.make_workload(cfg, 2)
    batches = [synth.make_batch(cfg, 50 + i) for i in range(4)]
    depths = [1, 1, 2, 2]
    # sequential reference
    ref = GpuStepper(cfg, w)
    ref_losses = []
    try:
        for (x, y), d in zip(batches, depths):
            ref.set_batch(x, y)
            ref_losses.append(ref.step(d, update=True))
        ref_p = {l: {k: ref.model.param(l, k).cpu() for k in synth.adapter_keys(cfg)}
                 for l in range(cfg.n_layers)}
    finally:
        ref.close()
    run = PrefixRun(cfg, w)
    try:
        A, Bs = torch.cuda.Stream(), torch.cuda.Stream()
        xs = [torch.tensor(x).to(run.x.dtype).cuda() for x, _ in batches]
        ys = [torch.tensor(y).cuda() for _, y in batches]
        losses = [torch.zeros(1, dtype=torch.float32, device="cuda") for _ in batches]
        done_prefix = [torch.cuda.Event() for _ in batches]
        done_suffix = [torch.cuda.Event() for _ in batches]
        torch.cuda.synchronize()
        R.ra_set_unfrozen_depth(run.ctx, depths[0])
        R.ra_forward_prefix(run.ctx, xs[0].data_ptr(), cfg.batch, cfg.seq, 0, stream=Bs.cuda_stream)
        done_prefix[0].record(Bs)
        for s in range(len(batches)):
            buf = s % 2
            A.wait_event(done_prefix[s])
            R.ra_forward_suffix(run.ctx, buf, ys[s].data_ptr(), losses[s].data_ptr(),
                                stream=A.cuda_stream)
            done_suffix[s].record(A)
            if s + 1 < len(batches):
                # the next batch's prefix at its own depth; it writes the other buffer, last
                # read by the suffix of step s - 1
                R.ra_set_unfrozen_depth(run.ctx, depths[s + 1])
                if s >= 1:
                    Bs.wait_event(done_suffix[s - 1])
                R.ra_forward_prefix(run.ctx, xs[s + 1].data_ptr(), cfg.batch, cfg.seq, 1 - buf,
                                    stream=Bs.cuda_stream)
                done_prefix[s + 1].record(Bs)
            R.ra_backward_truncated(run.ctx, cfg.n_layers - depths[s], stream=A.cuda_stream)
            R.ra_adapter_update(run.ctx, stream=A.cuda_stream)
        torch.cuda.synchronize()
        R.ra_sync_status(run.ctx)
        assert [l.item() for l in losses] == ref_losses
        for l in range(cfg.n_layers):
            for k in synth.adapter_keys(cfg):
                assert bool((run.model.param(l, k).cpu() == ref_p[l][k]).all()), (l, k)
    finally:
        run.close()


def test_split_calls_reject_out_of_order_use():
    cfg = synth.CONFIGS["tiny"]
    run = PrefixRun(cfg, synth.make_workload(cfg, 0))
    try:
        with pytest.raises(R.RingAdaError) as e:       # nothing in buffer 1 yet
            R.ra_forward_suffix(run.ctx, 1, run.labels.data_ptr(), run.loss.data_ptr())
        assert e.value.status == R.RA_ERR_STATE
        R.ra_set_unfrozen_depth(run.ctx, 1)
        R.ra_forward_prefix(run.ctx, run.x.data_ptr(), cfg.batch, cfg.seq, 1)
        R.ra_set_unfrozen_depth(run.ctx, 2)            # the prefix stops at the old depth
        with pytest.raises(R.RingAdaError) as e:
            R.ra_forward_suffix(run.ctx, 1, run.labels.data_ptr(), run.loss.data_ptr())
        assert e.value.status == R.RA_ERR_STATE
        with pytest.raises(R.RingAdaError) as e:
            R.ra_forward_prefix(run.ctx, run.x.data_ptr(), cfg.batch, cfg.seq, 2)
        assert e.value.status == R.RA_ERR_ARG
        R.ra_sync_status(run.ctx)
    finally:
        run.close()
    # a context without prefix buffers
    plain = GpuStepper(cfg, synth.make_workload(cfg, 0))
    try:
        with pytest.raises(R.RingAdaError) as e:
            R.ra_forward_prefix(plain.ctx, plain.x.data_ptr(), cfg.batch, cfg.seq, 0)
        assert e.value.status == R.RA_ERR_UNSUPPORTED
    finally:
        plain.close()
