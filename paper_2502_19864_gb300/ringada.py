"""ctypes binding of libringada (argument marshalling only; every step runs in the library).

The functions carry the C names (``ra_create``, ``ra_forward``, ...).  Each raises
``RingAdaError`` on a non-OK status, with the context's message.  ``Model`` is a small
convenience that lets PyTorch own the device buffers the library binds.
"""
from __future__ import annotations

import ctypes as C
import os
import re

import numpy as np

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libringada.so")
HEADER = os.path.join(os.path.dirname(PKG), "include", "ringada.h")

RA_OK, RA_ERR_ARG, RA_ERR_STATE, RA_ERR_NOT_SAVED, RA_ERR_SHAPE, RA_ERR_NOMEM, RA_ERR_CUDA, \
    RA_ERR_TIMEOUT, RA_ERR_UNSUPPORTED = range(9)
STATUS_NAMES = {0: "RA_OK", 1: "RA_ERR_ARG", 2: "RA_ERR_STATE", 3: "RA_ERR_NOT_SAVED",
                4: "RA_ERR_SHAPE", 5: "RA_ERR_NOMEM", 6: "RA_ERR_CUDA", 7: "RA_ERR_TIMEOUT",
                8: "RA_ERR_UNSUPPORTED"}
RA_ENCODER_POSTLN, RA_DECODER_PRENORM, RA_ENCODER_POSTLN_SPAN = 0, 1, 2
RA_F32, RA_BF16 = 0, 1
RA_ADAPTERS_HOULSBY, RA_ADAPTERS_POST_FFN = 0, 1

# ra_param ids (same order as the header's enum)
PARAMS = ["RA_P_WQKV", "RA_P_BQKV", "RA_P_WO", "RA_P_BO", "RA_P_LN1_G", "RA_P_LN1_B",
          "RA_P_W1", "RA_P_B1", "RA_P_W2", "RA_P_B2", "RA_P_LN2_G", "RA_P_LN2_B",
          "RA_P_WDA", "RA_P_WUA", "RA_P_WDF", "RA_P_WUF",
          "RA_P_WQ", "RA_P_WK", "RA_P_WV", "RA_P_RMS1_G", "RA_P_WG", "RA_P_WU", "RA_P_WD",
          "RA_P_RMS2_G", "RA_P_HEAD_W", "RA_P_HEAD_B", "RA_P_RMSF_G"]
P = {name: i for i, name in enumerate(PARAMS)}
# synthetic-workload key -> ra_param
KEY_TO_PARAM = {
    "Wqkv": "RA_P_WQKV", "bqkv": "RA_P_BQKV", "Wo": "RA_P_WO", "bo": "RA_P_BO",
    "ln1_g": "RA_P_LN1_G", "ln1_b": "RA_P_LN1_B", "W1": "RA_P_W1", "b1": "RA_P_B1",
    "W2": "RA_P_W2", "b2": "RA_P_B2", "ln2_g": "RA_P_LN2_G", "ln2_b": "RA_P_LN2_B",
    "WdA": "RA_P_WDA", "WuA": "RA_P_WUA", "WdF": "RA_P_WDF", "WuF": "RA_P_WUF",
    "Wq": "RA_P_WQ", "Wk": "RA_P_WK", "Wv": "RA_P_WV", "rms1_g": "RA_P_RMS1_G",
    "Wg": "RA_P_WG", "Wu": "RA_P_WU", "Wd": "RA_P_WD", "rms2_g": "RA_P_RMS2_G",
    "Wh": "RA_P_HEAD_W", "bh": "RA_P_HEAD_B", "rmsf_g": "RA_P_RMSF_G",
}


class ra_model_cfg(C.Structure):
    _fields_ = [("arch", C.c_int32), ("n_layers", C.c_int32), ("hidden", C.c_int32),
                ("n_heads", C.c_int32), ("ffn", C.c_int32), ("n_out", C.c_int32),
                ("max_batch", C.c_int32), ("max_seq", C.c_int32), ("dtype", C.c_int32),
                ("head_trainable", C.c_int32), ("max_depth", C.c_int32),
                ("norm_eps", C.c_float), ("rope_theta", C.c_float),
                ("adapter_placement", C.c_int32), ("prefix_buffers", C.c_int32)]


class ra_adam_cfg(C.Structure):
    _fields_ = [("lr", C.c_float), ("beta1", C.c_float), ("beta2", C.c_float), ("eps", C.c_float)]


class ra_tensor_desc(C.Structure):
    _fields_ = [("layer", C.c_int32), ("param", C.c_int32), ("data_dev", C.c_void_p),
                ("numel", C.c_int64)]


class ra_stats(C.Structure):
    _fields_ = [("weights_bytes", C.c_int64), ("trainable_bytes", C.c_int64),
                ("workspace_bytes", C.c_int64), ("saved_bytes_capacity", C.c_int64),
                ("saved_bytes_in_use", C.c_int64), ("depth", C.c_int32),
                ("k_forward", C.c_int32), ("k_backward", C.c_int32), ("n_updates", C.c_int32),
                ("tokens", C.c_int32), ("num_sms", C.c_int32)]


PROF_CATS = ["gemm", "attn_fwd", "attn_bwd", "adapter_fwd", "adapter_bwd", "norm", "head", "update"]


class ra_profile(C.Structure):
    _fields_ = [("ms", C.c_double * 8), ("flops", C.c_double * 8), ("bytes", C.c_double * 8),
                ("calls", C.c_int32 * 8)]


class ra_profile_record(C.Structure):
    _fields_ = [("cat", C.c_int32), ("ms", C.c_float), ("flops", C.c_double), ("bytes", C.c_double)]


class RingAdaError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__("%s: %s" % (STATUS_NAMES.get(status, status), msg))
        self.status = status


_lib = None

_SIGS = {
    "ra_create": (C.c_int, [C.POINTER(ra_model_cfg), C.c_int32, C.POINTER(C.c_void_p)]),
    "ra_required_bytes": (C.c_int, [C.c_void_p, C.POINTER(C.c_size_t), C.POINTER(C.c_size_t),
                                    C.POINTER(C.c_size_t)]),
    "ra_bind_memory": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p, C.c_size_t,
                                 C.c_void_p, C.c_size_t]),
    "ra_set_weights": (C.c_int, [C.c_void_p, C.POINTER(ra_tensor_desc), C.c_int32, C.c_void_p]),
    "ra_set_unfrozen_depth": (C.c_int, [C.c_void_p, C.c_int32]),
    "ra_schedule_depth": (C.c_int32, [C.c_int32, C.c_int32, C.c_int32, C.c_int32]),
    "ra_forward": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32, C.c_int32,
                             C.c_void_p, C.c_void_p, C.c_void_p]),
    "ra_forward_prefix": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_int32,
                                    C.c_void_p]),
    "ra_forward_suffix": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                    C.c_void_p]),
    "ra_backward_truncated": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p]),
    "ra_adapter_update": (C.c_int, [C.c_void_p, C.POINTER(ra_adam_cfg), C.c_void_p]),
    "ra_get_grad": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.POINTER(C.c_void_p),
                              C.POINTER(C.c_int64)]),
    "ra_get_param": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.POINTER(C.c_void_p),
                               C.POINTER(C.c_int64)]),
    "ra_trainable_state_bytes": (C.c_int, [C.c_void_p, C.POINTER(C.c_size_t)]),
    "ra_get_trainable": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t]),
    "ra_set_trainable": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t]),
    "ra_get_stats": (C.c_int, [C.c_void_p, C.POINTER(ra_stats)]),
    "ra_sync_status": (C.c_int, [C.c_void_p, C.c_void_p]),
    "ra_last_error": (C.c_char_p, [C.c_void_p]),
    "ra_selftest_wait_timeout": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p]),
    "ra_eval_activation": (C.c_int, [C.c_int32, C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p]),
    "ra_destroy": (None, [C.c_void_p]),
    "ra_gemm_bf16": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32, C.c_int32,
                               C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p]),
    "ra_gemm_bf16_epi": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_int32,
                                   C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32,
                                   C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p]),
    "ra_gemm_scratch_bytes": (C.c_size_t, []),
    "ra_adapter_backward": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                      C.c_int32, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p,
                                      C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p]),
    "ra_adapter_backward_scratch_bytes": (C.c_size_t, [C.c_int32, C.c_int32, C.c_int32]),
    "ra_adapter_backward_noalloc": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                              C.c_void_p, C.c_int32, C.c_int32, C.c_int32,
                                              C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "ra_adapter_backward_noalloc_capacity": (C.c_size_t, []),
    "ra_profile_enable": (C.c_int, [C.c_void_p, C.c_int32]),
    "ra_profile_read": (C.c_int, [C.c_void_p, C.c_void_p]),
    "ra_kernel_launches": (C.c_int64, []),
    "ra_profile_gemm_log": (C.c_int, [C.c_void_p, C.c_int32]),
    "ra_profile_gemm_replay": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32), C.POINTER(C.c_double),
                                         C.c_void_p]),
    "ra_profile_records": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.POINTER(C.c_int32)]),
}


def header_functions():
    """Names of the functions include/ringada.h declares."""
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ra_[a-z0-9_]+)\s*\(", text)))


def lib():
    """Loads libringada.so; raises if it has not been built (there is no other path)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libringada.so is missing: build it with __graft_entry__.build()")
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _check(status, ctx=None):
    if status != RA_OK:
        msg = lib().ra_last_error(ctx).decode() if ctx else ""
        raise RingAdaError(status, msg)


def _stream_ptr(stream):
    if stream is None:
        return None
    return C.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


# ---- thin wrappers with the C names ---------------------------------------------------------

def ra_create(cfg: ra_model_cfg, adapter_dim: int):
    h = C.c_void_p()
    _check(lib().ra_create(C.byref(cfg), adapter_dim, C.byref(h)))
    return h


def ra_required_bytes(ctx):
    w, t, s = C.c_size_t(), C.c_size_t(), C.c_size_t()
    _check(lib().ra_required_bytes(ctx, C.byref(w), C.byref(t), C.byref(s)), ctx)
    return w.value, t.value, s.value


def ra_bind_memory(ctx, w_ptr, w_bytes, t_ptr, t_bytes, s_ptr, s_bytes):
    _check(lib().ra_bind_memory(ctx, w_ptr, w_bytes, t_ptr, t_bytes, s_ptr, s_bytes), ctx)


def ra_set_weights(ctx, descs, stream=None):
    arr = (ra_tensor_desc * len(descs))(*descs)
    _check(lib().ra_set_weights(ctx, arr, len(descs), _stream_ptr(stream)), ctx)


def ra_set_unfrozen_depth(ctx, d: int):
    _check(lib().ra_set_unfrozen_depth(ctx, d), ctx)


def ra_forward(ctx, x_ptr, labels_ptr, B, S, loss_ptr, logits_ptr=None, stream=None):
    _check(lib().ra_forward(ctx, x_ptr, labels_ptr, B, S, loss_ptr, logits_ptr,
                            _stream_ptr(stream)), ctx)


def ra_forward_prefix(ctx, x_ptr, B, S, buf, stream=None):
    _check(lib().ra_forward_prefix(ctx, x_ptr, B, S, buf, _stream_ptr(stream)), ctx)


def ra_forward_suffix(ctx, buf, labels_ptr, loss_ptr, logits_ptr=None, stream=None):
    _check(lib().ra_forward_suffix(ctx, buf, labels_ptr, loss_ptr, logits_ptr,
                                   _stream_ptr(stream)), ctx)


def ra_backward_truncated(ctx, k: int, stream=None):
    _check(lib().ra_backward_truncated(ctx, k, _stream_ptr(stream)), ctx)


def ra_adapter_update(ctx, lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8, stream=None):
    a = ra_adam_cfg(lr, beta1, beta2, eps)
    _check(lib().ra_adapter_update(ctx, C.byref(a), _stream_ptr(stream)), ctx)


def ra_get_grad(ctx, layer, which):
    p, n = C.c_void_p(), C.c_int64()
    _check(lib().ra_get_grad(ctx, layer, which, C.byref(p), C.byref(n)), ctx)
    return p.value, n.value


def ra_get_param(ctx, layer, which):
    p, n = C.c_void_p(), C.c_int64()
    _check(lib().ra_get_param(ctx, layer, which, C.byref(p), C.byref(n)), ctx)
    return p.value, n.value


def ra_trainable_state_bytes(ctx):
    n = C.c_size_t()
    _check(lib().ra_trainable_state_bytes(ctx, C.byref(n)), ctx)
    return n.value


def ra_get_trainable(ctx):
    n = ra_trainable_state_bytes(ctx)
    buf = np.empty(n, dtype=np.uint8)
    _check(lib().ra_get_trainable(ctx, buf.ctypes.data, n), ctx)
    return buf


def ra_set_trainable(ctx, blob: np.ndarray):
    blob = np.ascontiguousarray(blob, dtype=np.uint8)
    _check(lib().ra_set_trainable(ctx, blob.ctypes.data, blob.nbytes), ctx)


def ra_get_stats(ctx):
    s = ra_stats()
    _check(lib().ra_get_stats(ctx, C.byref(s)), ctx)
    return {name: getattr(s, name) for name, _ in ra_stats._fields_}


def ra_sync_status(ctx, stream=None):
    _check(lib().ra_sync_status(ctx, _stream_ptr(stream)), ctx)


def ra_selftest_wait_timeout(ctx, limit_us: int, stream=None):
    _check(lib().ra_selftest_wait_timeout(ctx, limit_us, _stream_ptr(stream)), ctx)


def ra_eval_activation(which: int, x_ptr, y_ptr, n: int, stream=None):
    _check(lib().ra_eval_activation(which, x_ptr, y_ptr, n, _stream_ptr(stream)))


def ra_last_error(ctx) -> str:
    return lib().ra_last_error(ctx).decode()


def ra_destroy(ctx):
    lib().ra_destroy(ctx)


def ra_gemm_bf16(A_ptr, B_ptr, C_ptr, M, N, K, bias_ptr=None, gelu_ptr=None, stream=None):
    _check(lib().ra_gemm_bf16(A_ptr, B_ptr, C_ptr, M, N, K, bias_ptr, gelu_ptr, _stream_ptr(stream)))


RA_EPI_STORE, RA_EPI_BIAS_GELU, RA_EPI_MUL, RA_EPI_RESID, RA_EPI_BIAS_GELU_G = 0, 1, 2, 3, 6
RA_EPI_B_KN = 0x100


def ra_gemm_scratch_bytes() -> int:
    return int(lib().ra_gemm_scratch_bytes())


def ra_gemm_bf16_epi(A_ptr, B_ptr, M, N, K, epi, bias_ptr=None, aux_ptr=None, C_ptr=None,
                     c_dtype=RA_BF16, C2_ptr=None, scratch_ptr=None, scratch_bytes=0, stream=None):
    _check(lib().ra_gemm_bf16_epi(A_ptr, B_ptr, M, N, K, epi, bias_ptr, aux_ptr, C_ptr, c_dtype,
                                  C2_ptr, scratch_ptr, scratch_bytes, _stream_ptr(stream)))


def ra_adapter_backward_scratch_bytes(T, H, m) -> int:
    return lib().ra_adapter_backward_scratch_bytes(T, H, m)


def ra_adapter_backward(g, h, z, Wd, Wu, T, H, m, dWd, dWu, dh, scratch, scratch_bytes, stream=None):
    _check(lib().ra_adapter_backward(g, h, z, Wd, Wu, T, H, m, dWd, dWu, dh, scratch,
                                     scratch_bytes, _stream_ptr(stream)))


def ra_adapter_backward_noalloc(g, h, z, Wd, Wu, T, H, m, dWd, dWu, dh, stream=None):
    """The adapter backward with the library's fixed scratch array (no allocation)."""
    _check(lib().ra_adapter_backward_noalloc(g, h, z, Wd, Wu, T, H, m, dWd, dWu, dh,
                                             _stream_ptr(stream)))


def ra_adapter_backward_noalloc_capacity() -> int:
    return lib().ra_adapter_backward_noalloc_capacity()


def ra_profile_enable(ctx, on: bool):
    _check(lib().ra_profile_enable(ctx, 1 if on else 0), ctx)


def ra_profile_read(ctx):
    """Per-category {ms, flops, bytes, calls} of the recorded kernel calls."""
    p = ra_profile()
    _check(lib().ra_profile_read(ctx, C.byref(p)), ctx)
    return {cat: dict(ms=p.ms[i], flops=p.flops[i], bytes=p.bytes[i], calls=p.calls[i])
            for i, cat in enumerate(PROF_CATS)}


def ra_profile_records(ctx, max_records=4096):
    """[(category, ms, flops, bytes)] of every recorded kernel call, in call order."""
    arr = (ra_profile_record * max_records)()
    n = C.c_int32()
    _check(lib().ra_profile_records(ctx, arr, max_records, C.byref(n)), ctx)
    return [(PROF_CATS[r.cat], r.ms, r.flops, r.bytes) for r in arr[:min(n.value, max_records)]]


def ra_profile_gemm_log(ctx, on: bool):
    _check(lib().ra_profile_gemm_log(ctx, 1 if on else 0), ctx)


def ra_profile_gemm_replay(ctx, stream=None):
    """Re-launches the recorded GEMMs back to back; returns (launches, flops)."""
    n, fl = C.c_int32(), C.c_double()
    _check(lib().ra_profile_gemm_replay(ctx, C.byref(n), C.byref(fl), _stream_ptr(stream)), ctx)
    return n.value, fl.value


def ra_kernel_launches() -> int:
    return lib().ra_kernel_launches()


# ---- convenience: torch-owned buffers ------------------------------------------------------

def schedule_depth(step_index: int, interval: int = 50, d0: int = 1, d_max: int = 12) -> int:
    """Top-down unfreezing (Algorithm 1: d <- d + 1 every interval), per 0-based step."""
    d = lib().ra_schedule_depth(step_index, interval, d0, d_max)
    if d < 0:
        raise RingAdaError(RA_ERR_ARG, "ra_schedule_depth: invalid arguments")
    return d


def make_cfg(arch, n_layers, hidden, n_heads, ffn, n_out, max_batch, max_seq, dtype,
             head_trainable, max_depth=0, norm_eps=1e-12, rope_theta=10000.0,
             adapter_placement=0, prefix_buffers=0):
    return ra_model_cfg(arch, n_layers, hidden, n_heads, ffn, n_out, max_batch, max_seq, dtype,
                        head_trainable, max_depth, norm_eps, rope_theta, adapter_placement,
                        prefix_buffers)


class Model:
    """A context plus PyTorch-allocated device buffers (weights, trainable, workspace)."""

    def __init__(self, cfg: ra_model_cfg, adapter_dim: int, device="cuda"):
        import torch
        self.torch = torch
        self.cfg = cfg
        self.ctx = ra_create(cfg, adapter_dim)
        w, t, s = ra_required_bytes(self.ctx)
        self.buffers = [torch.empty(max(n, 256), dtype=torch.uint8, device=device) for n in (w, t, s)]
        ptrs = [b.data_ptr() for b in self.buffers]
        ra_bind_memory(self.ctx, ptrs[0], self.buffers[0].numel(), ptrs[1],
                       self.buffers[1].numel(), ptrs[2], self.buffers[2].numel())
        self.device = device

    def set_weights(self, layers, head, stream=None):
        """layers: list of {key: array}; head: {key: array} (synthetic-workload keys)."""
        torch = self.torch
        keep, descs = [], []
        for l, p in enumerate(layers):
            for key, arr in p.items():
                t = torch.as_tensor(np.ascontiguousarray(arr, dtype=np.float32)).to(self.device)
                keep.append(t)
                descs.append(ra_tensor_desc(l, P[KEY_TO_PARAM[key]], t.data_ptr(), t.numel()))
        for key, arr in head.items():
            t = torch.as_tensor(np.ascontiguousarray(arr, dtype=np.float32)).to(self.device)
            keep.append(t)
            descs.append(ra_tensor_desc(-1, P[KEY_TO_PARAM[key]], t.data_ptr(), t.numel()))
        ra_set_weights(self.ctx, descs, stream)
        torch.cuda.synchronize()

    def grad(self, layer, key):
        ptr, n = ra_get_grad(self.ctx, layer, P[KEY_TO_PARAM[key]])
        return self._view(ptr, n)

    def param(self, layer, key):
        ptr, n = ra_get_param(self.ctx, layer, P[KEY_TO_PARAM[key]])
        return self._view(ptr, n)

    def _view(self, ptr, n):
        """Copy of a float32 device range [ptr, ptr + 4n) as a torch tensor."""
        torch = self.torch
        base = self.buffers[1]
        off = ptr - base.data_ptr()
        assert 0 <= off and off + 4 * n <= base.numel()
        return base[off:off + 4 * n].view(torch.float32).clone()

    def stats(self):
        return ra_get_stats(self.ctx)

    def close(self):
        if self.ctx is not None:
            ra_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
