"""The feed-forward units' GELU on the device (both paths), against float64.

The denoiser's FFN applies GELU in its erf form, x Phi(x) (the transformer of
Sec. 3.1).  The kernels evaluate erf with Abramowitz & Stegun's formula 7.1.26,
whose absolute error is at most 1.5e-7; evo_test_gelu runs that same device
function on a dense grid and on special values.  The bound below is the
formula's error scaled by x/2, plus the fp32 rounding of the exponential's
argument (relative, proportional to erfc) and of the result.
"""
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu


def _exact(x64):
    return 0.5 * x64 * (1.0 + torch.special.erf(x64 / math.sqrt(2.0)))


@pytest.mark.parametrize("packed", [False, True])
def test_gelu_within_the_published_bound(packed):
    from paper_2607_20293_gb300 import binding
    x = torch.linspace(-16.0, 16.0, 4_000_001, dtype=torch.float32)
    rng = np.random.default_rng(11)
    extra = torch.from_numpy(rng.standard_normal(1_000_000).astype(np.float32) * 3.0)
    x = torch.cat([x, extra])
    y = binding.test_gelu(x.cuda(), packed=packed).cpu().double()
    x64 = x.double()
    ref = _exact(x64)
    erfc = torch.special.erfc(x64.abs() / math.sqrt(2.0))
    bound = 0.5 * x64.abs() * (1.6e-7 + 4e-6 * erfc) + 2.0 ** -22 * ref.abs() + 1e-37
    err = (y - ref).abs()
    worst = int(torch.argmax(err / bound))
    assert bool((err <= bound).all()), f"x {x64[worst].item()} y {y[worst].item()} exact {ref[worst].item()}"
    # the large-|x| limits hold exactly in fp32
    big = x64.abs() >= 8
    assert bool((y[big & (x64 > 0)] == x64[big & (x64 > 0)]).all())
    assert bool((y[big & (x64 < 0)].abs() <= 1e-13).all())


@pytest.mark.parametrize("packed", [False, True])
def test_gelu_special_values(packed):
    from paper_2607_20293_gb300 import binding
    x = torch.tensor([0.0, -0.0, float("inf"), float("-inf"), float("nan"), 1e-30, -1e-30, 3e38, -3e38, 0.5],
                     dtype=torch.float32)
    y = binding.test_gelu(x.cuda(), packed=packed).cpu()
    assert y[0].item() == 0.0 and y[1].item() == 0.0
    assert y[2].item() == float("inf")
    assert y[3].item() == 0.0
    assert math.isnan(y[4].item())
    assert abs(y[5].item() - 0.5e-30) <= 1e-36 and abs(y[6].item() + 0.5e-30) <= 1e-36
    assert y[7].item() == pytest.approx(3e38, rel=1e-7)
    assert y[8].item() == 0.0


def test_packed_and_scalar_forms_agree_bitwise():
    from paper_2607_20293_gb300 import binding
    rng = np.random.default_rng(5)
    x = torch.from_numpy((rng.standard_normal(2_000_001) * 4.0).astype(np.float32)).cuda()
    a = binding.test_gelu(x, packed=False)
    b = binding.test_gelu(x, packed=True)
    diff = (a.view(torch.int32) != b.view(torch.int32)).nonzero().flatten()[:5].tolist()
    assert not diff, [(x[i].item(), a[i].item(), b[i].item()) for i in diff]


def test_gelu_rejects_host_pointers_and_negative_sizes():
    from paper_2607_20293_gb300 import binding
    lib = binding.load()
    x = torch.zeros(4, dtype=torch.float32)
    assert lib.evo_test_gelu(x.data_ptr(), x.data_ptr(), 4, 0, None) == binding.ERR_ARG
    xc = x.cuda()
    assert lib.evo_test_gelu(xc.data_ptr(), xc.data_ptr(), -1, 0, None) == binding.ERR_ARG
    assert lib.evo_test_gelu(xc.data_ptr(), xc.data_ptr(), 4, 2, None) == binding.ERR_ARG
    assert lib.evo_test_gelu(xc.data_ptr(), xc.data_ptr(), 0, 1, None) == binding.OK
