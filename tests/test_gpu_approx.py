"""The hardware approximations behind the step kernel's certified fast path
(sqrt.approx.f32, div.approx.f32) stay far inside the 2^-19 relative error
the certificate assumes, over operands spanning the ranges the update sees
(denominators in [2^-125, 2^125], numerators of any magnitude)."""
import ctypes
import subprocess
from pathlib import Path

import pytest
import torch

pytestmark = pytest.mark.gpu
HERE = Path(__file__).resolve().parent


@pytest.fixture(scope="module")
def probe(tmp_path_factory):
    out = tmp_path_factory.mktemp("approx") / "libapprox_probe.so"
    subprocess.run(["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "--ftz=false",
                    "-Xcompiler", "-fPIC", "-shared", str(HERE / "cuda" / "approx_probe.cu"), "-o", str(out)],
                   check=True)
    lib = ctypes.CDLL(str(out))
    lib.approx_probe.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]
    return lib


def test_approximations_within_certificate_bound(probe):
    g = torch.Generator(device="cuda").manual_seed(0)
    n = 1 << 26
    worst = []
    for lo, hi in [(-125, 125), (-30, 30), (-2, 2)]:
        ea = torch.randint(-126, 127, (n,), device="cuda", generator=g).float()
        eb = torch.randint(lo, hi, (n,), device="cuda", generator=g).float()
        a = (torch.rand(n, device="cuda", generator=g) + 1) * torch.exp2(ea) * torch.sign(torch.randn(n, device="cuda", generator=g))
        b = (torch.rand(n, device="cuda", generator=g) + 1) * torch.exp2(eb)
        out = torch.zeros(2, device="cuda")
        assert probe.approx_probe(a.data_ptr(), b.data_ptr(), n, out.data_ptr()) == 0
        worst.append(out.cpu().tolist())
    for s_err, d_err in worst:
        assert s_err < 2.0 ** -21, s_err
        assert d_err < 2.0 ** -21, d_err
