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
    # adapter placement: Houlsby or the paper's post-FFN adapter (encoders only)
    with pytest.raises(R.RingAdaError) as e:
        R.ra_create(enc_cfg(adapter_placement=5), 16)
    assert e.value.status == R.RA_ERR_ARG
    with pytest.raises(R.RingAdaError) as e:
        R.ra_create(enc_cfg(arch=R.RA_DECODER_PRENORM, n_out=64, head_trainable=0,
                            adapter_placement=R.RA_ADAPTERS_POST_FFN), 16)
    assert e.value.status == R.RA_ERR_SHAPE
    for arch in (R.RA_ENCODER_POSTLN, R.RA_ENCODER_POSTLN_SPAN):
        R.ra_destroy(R.ra_create(enc_cfg(arch=arch, adapter_placement=R.RA_ADAPTERS_POST_FFN), 16))
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


def test_schedule_depth_follows_the_unfreezing_rule(lib):
    # Algorithm 1 / the sched workload: d = min(1 + floor(s / 50), 12), evaluated in the
    # library (ra_schedule_depth)
    assert [R.schedule_depth(s) for s in (0, 49, 50, 99, 100, 549, 550, 599)] == \
        [1, 1, 2, 2, 3, 11, 12, 12]
    assert R.schedule_depth(7, interval=3, d0=2, d_max=4) == 4
    assert R.schedule_depth(0, interval=40, d0=1, d_max=24) == 1
    assert lib.ra_schedule_depth(-1, 50, 1, 12) == -1      # invalid arguments
    assert lib.ra_schedule_depth(5, 0, 1, 12) == -1


def _mb_set(sizes):
    # every buffer of the plan starts on a 256-byte boundary
    return sum((s + 255) // 256 * 256 for s in sizes)


@pytest.mark.parametrize("arch", ["encoder", "decoder", "post_ffn"])
def test_saved_set_per_layer_is_the_backward_inputs(lib, arch):
    """The activation arena holds, per unfrozen layer, exactly what the backward reads: the
    lowest layer k keeps the adapter and norm inputs of its FFN half and the A adapter's
    inputs (no attention backward runs there); every layer above also keeps q|k|v, the
    attention output and the row log-sum-exp (and, decoder, its fp32 input and RMS scale).
    With the paper's single post-FFN adapter the lowest layer keeps only that adapter's
    input and bottleneck pre-activation, and the layers above add both norms' xhat and
    rstd and GELU'(u).  Capacity = max_depth x the full set."""
    B, S, H, heads, F, m = 4, 64, 256, 4, 1024, 32
    T = B * S
    es = 2  # bf16
    if arch == "encoder":
        cfg = dict(arch=R.RA_ENCODER_POSTLN, n_out=2)
        lowest = [T * H * es, T * m * 4, T * H * es, T * 4, T * F * es, T * H * es, T * m * 4,
                  T * H * es, T * 4]          # a, zA, xhat1, rstd1, GELU'(u), f, zF, xhat2, rstd2
        full_only = [T * 3 * H * es, T * H * es, B * heads * S * 4]   # qkv, O, lse
    elif arch == "post_ffn":
        cfg = dict(arch=R.RA_ENCODER_POSTLN, n_out=2, adapter_placement=R.RA_ADAPTERS_POST_FFN)
        lowest = [T * H * es, T * m * 4]     # y2 (the adapter input), zF
        full_only = [T * 3 * H * es, T * H * es, B * heads * S * 4, T * H * es, T * 4,
                     T * F * es, T * H * es, T * 4]
        #            qkv, O, lse, xhat1, rstd1, GELU'(u), xhat2, rstd2
    else:
        cfg = dict(arch=R.RA_DECODER_PRENORM, n_out=64, head_trainable=0)
        lowest = [T * H * es, T * m * 4, T * H * 4, T * 4, T * 2 * F * es, T * H * es, T * m * 4]
        #         a, zA, x1 (f32), rstd2, gate|up, f, zF
        full_only = [T * H * 4, T * 4, T * 3 * H * es, T * H * es, B * heads * S * 4]
        #            x_in (f32), rstd1, qkv, O, lse
    full = _mb_set(lowest) + _mb_set(full_only)
    caps = []
    for md in (1, 3):
        ctx = R.ra_create(enc_cfg(n_layers=3, hidden=H, n_heads=heads, ffn=F, max_batch=B,
                                  max_seq=S, dtype=R.RA_BF16, max_depth=md, **cfg), m)
        caps.append(R.ra_get_stats(ctx)["saved_bytes_capacity"])
        R.ra_destroy(ctx)
    assert caps == [full, 3 * full]
