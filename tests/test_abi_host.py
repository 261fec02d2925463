"""Host-only checks of the C ABI: the library loads, exports what the header declares, and
validates arguments and call order without touching a GPU."""
import ctypes as C

import pytest

from paper_2502_19864_gb300 import ringada as R


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__.build()
    return R.lib()


def enc_cfg(**kw):
    base = dict(arch=R.RA_ENCODER_POSTLN, n_layers=4, hidden=128, n_heads=2, ffn=512, n_out=2,
                max_batch=4, max_seq=32, dtype=R.RA_F32, head_trainable=1, max_depth=0)
    base.update(kw)
    return R.make_cfg(**base)


def test_every_header_symbol_is_exported(lib):
    names = R.header_functions()
    assert "ra_create" in names and "ra_backward_truncated" in names
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing
    # and the binding covers every one of them
    assert sorted(R._SIGS) == names


def test_create_validates_shapes(lib):
    with pytest.raises(R.RingAdaError) as e:
        R.ra_create(enc_cfg(), 7)          # bottleneck not a multiple of 8
    assert e.value.status == R.RA_ERR_SHAPE
    with pytest.raises(R.RingAdaError) as e:
        R.ra_create(enc_cfg(hidden=96), 16)
    assert e.value.status == R.RA_ERR_SHAPE
    with pytest.raises(R.RingAdaError) as e:
        R.ra_create(enc_cfg(max_depth=9), 16)
    assert e.value.status == R.RA_ERR_ARG
    with pytest.raises(R.RingAdaError) as e:
        R.ra_create(enc_cfg(arch=7), 16)
    assert e.value.status == R.RA_ERR_ARG
    with pytest.raises(R.RingAdaError):   # decoder head must be frozen
        R.ra_create(enc_cfg(arch=R.RA_DECODER_PRENORM, n_out=64, head_trainable=1), 16)
    # the span head has exactly two outputs (start, end) and sequences of at most 4096
    for bad in (dict(n_out=3), dict(n_out=2, max_seq=4097)):
        with pytest.raises(R.RingAdaError) as e:
            R.ra_create(enc_cfg(arch=R.RA_ENCODER_POSTLN_SPAN, **bad), 16)
        assert e.value.status == R.RA_ERR_SHAPE
    R.ra_destroy(R.ra_create(enc_cfg(arch=R.RA_ENCODER_POSTLN_SPAN, n_out=2), 16))
    ctx = R.ra_create(enc_cfg(), 16)
    R.ra_destroy(ctx)


def test_required_bytes_shrink_with_max_depth(lib):
    sizes = []
    for md in (1, 2, 4):
        ctx = R.ra_create(enc_cfg(max_depth=md), 16)
        sizes.append(R.ra_required_bytes(ctx))
        st = R.ra_get_stats(ctx)
        R.ra_destroy(ctx)
        assert st["saved_bytes_capacity"] > 0 and st["depth"] == md
    assert sizes[0][0] == sizes[1][0] == sizes[2][0]      # weights independent of depth
    assert sizes[0][2] < sizes[1][2] < sizes[2][2]        # workspace grows with the arena
    per_layer = sizes[1][2] - sizes[0][2]
    assert sizes[2][2] - sizes[1][2] == 2 * per_layer


def test_depth_and_call_order_errors(lib):
    ctx = R.ra_create(enc_cfg(max_depth=3), 16)
    try:
        with pytest.raises(R.RingAdaError) as e:
            R.ra_set_unfrozen_depth(ctx, 0)
        assert e.value.status == R.RA_ERR_ARG
        with pytest.raises(R.RingAdaError) as e:
            R.ra_set_unfrozen_depth(ctx, 4)     # beyond max_depth
        assert e.value.status == R.RA_ERR_ARG
        assert "max_depth" in R.ra_last_error(ctx)
        R.ra_set_unfrozen_depth(ctx, 2)
        # nothing bound yet
        with pytest.raises(R.RingAdaError) as e:
            R.ra_forward(ctx, 16, 16, 1, 1, 16)
        assert e.value.status == R.RA_ERR_STATE
        with pytest.raises(R.RingAdaError) as e:
            R.ra_backward_truncated(ctx, 3)
        assert e.value.status == R.RA_ERR_STATE
        with pytest.raises(R.RingAdaError) as e:
            R.ra_adapter_update(ctx)
        assert e.value.status == R.RA_ERR_STATE
        with pytest.raises(R.RingAdaError) as e:
            R.ra_set_weights(ctx, [])
        assert e.value.status == R.RA_ERR_STATE
        with pytest.raises(R.RingAdaError) as e:
            R.ra_get_grad(ctx, 0, R.P["RA_P_WDA"])
        assert e.value.status == R.RA_ERR_STATE
    finally:
        R.ra_destroy(ctx)


def test_bind_checks_sizes_and_alignment_before_the_device(lib):
    ctx = R.ra_create(enc_cfg(), 16)
    try:
        w, t, s = R.ra_required_bytes(ctx)
        with pytest.raises(R.RingAdaError) as e:
            R.ra_bind_memory(ctx, 256, w - 1, 512, t, 768, s)
        assert e.value.status == R.RA_ERR_NOMEM
        with pytest.raises(R.RingAdaError) as e:
            R.ra_bind_memory(ctx, 260, w, 512, t, 768, s)
        assert e.value.status == R.RA_ERR_ARG
        with pytest.raises(R.RingAdaError) as e:
            R.ra_bind_memory(ctx, None, w, 512, t, 768, s)
        assert e.value.status == R.RA_ERR_ARG
    finally:
        R.ra_destroy(ctx)


def test_null_arguments_are_rejected(lib):
    assert lib.ra_create(None, 16, C.byref(C.c_void_p())) == R.RA_ERR_ARG
    assert lib.ra_get_stats(None, None) == R.RA_ERR_ARG
    assert lib.ra_last_error(None) == b"null context"
    lib.ra_destroy(None)
    assert lib.ra_adapter_backward_scratch_bytes(0, 16, 16) == 0
    assert lib.ra_adapter_backward_scratch_bytes(128, 128, 16) > 128 * 16 * 4
    assert lib.ra_gemm_bf16(None, None, None, 1, 8, 8, None, None, None) == R.RA_ERR_ARG
    assert lib.ra_gemm_bf16(16, 16, 16, 1, 8, 12, None, None, None) == R.RA_ERR_SHAPE


def test_schedule_depth_follows_the_unfreezing_rule():
    # Algorithm 1 / the sched workload: d = min(1 + floor(s / 50), 12)
    assert [R.schedule_depth(s) for s in (0, 49, 50, 99, 100, 549, 550, 599)] == \
        [1, 1, 2, 2, 3, 11, 12, 12]
