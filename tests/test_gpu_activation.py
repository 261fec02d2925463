"""The step's activation code (ra_eval_activation) against the exact functions in fp64.

GELU and GELU' are evaluated in the kernels with erf from Abramowitz & Stegun formula
7.1.28, whose published absolute error bound is 3e-7; evaluated in fp32 (without
cancellation) it stays within 4.5e-7.  The bounds below carry that through
GELU(x) = x (1 + erf(x / sqrt 2)) / 2 and GELU'(x) = Phi(x) + x phi(x), plus fp32 rounding.
SiLU and its derivative are checked at fp32 accuracy."""
import numpy as np
import pytest
from scipy.special import erf

from paper_2502_19864_gb300 import ringada as R

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


def _eval(which, x):
    import torch
    xd = torch.tensor(x, dtype=torch.float32, device="cuda")
    yd = torch.full_like(xd, float("nan"))
    R.ra_eval_activation(which, xd.data_ptr(), yd.data_ptr(), xd.numel())
    torch.cuda.synchronize()
    return yd.cpu().numpy().astype(np.float64)


def _grid():
    x = np.concatenate([np.linspace(-12.0, 12.0, 480001), np.array([0.0, -0.0, 1e-30, -1e-30, 1e-8, -1e-8,
                                                                    40.0, -40.0, 1e4, -1e4, 3e38, -3e38])])
    return x.astype(np.float32).astype(np.float64)  # the values the kernel sees


def test_gelu_within_the_published_erf_bound():
    x = _grid()
    y = _eval(0, x)
    ref = 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))
    err = np.abs(y - ref)
    bound = 0.5 * np.abs(x) * 4.5e-7 + 2.5e-7 * np.abs(ref) + 1e-37
    assert np.all(np.isfinite(y))
    worst = int(np.argmax(err / bound))
    assert np.all(err <= bound), (x[worst], y[worst], ref[worst])


def test_gelu_grad_within_the_published_erf_bound():
    x = _grid()
    x = x[np.abs(x) < 1e3]  # x phi(x) underflows far out; the large values are covered above
    y = _eval(1, x)
    phi = np.exp(-0.5 * x * x) / np.sqrt(2.0 * np.pi)
    ref = 0.5 * (1.0 + erf(x / np.sqrt(2.0))) + x * phi
    err = np.abs(y - ref)
    bound = 0.5 * 4.5e-7 + 2.5e-7 * np.abs(ref) + 1e-6 * np.abs(x * phi) * (1.0 + 0.5 * x * x)
    worst = int(np.argmax(err / bound))
    assert np.all(err <= bound), (x[worst], y[worst], ref[worst])


def test_silu_and_its_derivative():
    x = np.linspace(-30.0, 30.0, 120001).astype(np.float32).astype(np.float64)
    s = 1.0 / (1.0 + np.exp(-x))
    for which, ref in ((2, x * s), (3, s * (1.0 + x * (1.0 - s)))):
        y = _eval(which, x)
        err = np.abs(y - ref)
        assert np.all(err <= 1e-6 * np.maximum(1.0, np.abs(ref))), which


def test_bad_selector_is_rejected():
    with pytest.raises(R.RingAdaError):
        R.ra_eval_activation(7, None, None, 0)
