"""Host-side checks of the C ABI (no GPU): the library loads, exports every
symbol include/tq.h declares, and rejects bad arguments before touching a device."""
import ctypes
import os
import re

import pytest

from paper_2606_18114_gb300 import build as tqbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    path = tqbuild.build()
    from paper_2606_18114_gb300 import tq
    return tq.load(path)


def _declared():
    with open(os.path.join(ROOT, "include", "tq.h")) as f:
        text = f.read()
    return re.findall(r"TQ_API\s+[\w\s\*]+?\b(tq_\w+)\s*\(", text)


def test_header_declares_expected_symbols():
    from paper_2606_18114_gb300 import tq
    assert sorted(_declared()) == sorted(tq.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_exports_are_exactly_the_header(lib):
    import subprocess
    out = subprocess.run(["nm", "-D", "--defined-only", lib._name], capture_output=True, text=True)
    if out.returncode != 0:
        pytest.skip("nm unavailable")
    tq_syms = sorted(set(re.findall(r"\b(tq_\w+)\b", out.stdout)))
    assert tq_syms == sorted(_declared())


def test_version_and_empty_error(lib):
    assert b"sm_103a" in lib.tq_version()
    assert lib.tq_last_error() is not None


def test_missing_library_fails_loudly(tmp_path):
    from paper_2606_18114_gb300 import tq
    saved = tq._lib
    tq._lib = None
    try:
        with pytest.raises(RuntimeError):
            tq.load(str(tmp_path / "nope.so"))
    finally:
        tq._lib = saved


FAKE = 1 << 20  # aligned, never dereferenced: every call below fails validation first
MIS = FAKE + 4  # misaligned


@pytest.mark.parametrize("args,status", [
    ((FAKE, 8, 256, 33, FAKE, FAKE, FAKE, None), 1),   # bad group size
    ((FAKE, 8, 200, 32, FAKE, FAKE, FAKE, None), 1),   # k % 16
    ((FAKE, 8, 96, 64, FAKE, FAKE, FAKE, None), 1),    # k % g
    ((FAKE, -1, 256, 32, FAKE, FAKE, FAKE, None), 1),  # negative
    ((None, 8, 256, 32, FAKE, FAKE, FAKE, None), 1),   # null w
    ((MIS, 8, 256, 32, FAKE, FAKE, FAKE, None), 1),    # misaligned w
    ((FAKE, 8, 256, 32, FAKE, None, FAKE, None), 1),   # null scales
    ((None, 0, 256, 32, None, None, None, None), 0),   # empty: nothing to do
    ((None, 8, 0, 32, None, None, None, None), 0),
])
def test_quantize_rejects_before_launch(lib, args, status):
    assert lib.tq_quantize(*args) == status
    if status:
        assert lib.tq_last_error()


@pytest.mark.parametrize("args,status", [
    ((FAKE, 4, 256, FAKE, FAKE, 64, 48, FAKE, 0, None), 1),    # bad group
    ((FAKE, 4, 96, FAKE, FAKE, 64, 32, FAKE, 0, None), 2),     # k % 64 unsupported
    ((FAKE, 4, 256, FAKE, FAKE, 64, 512, FAKE, 0, None), 1),   # k % g
    ((FAKE, 4, 256, FAKE, FAKE, 64, 32, FAKE, 7, None), 1),    # bad dtype
    ((None, 4, 256, FAKE, FAKE, 64, 32, FAKE, 0, None), 1),    # null x
    ((FAKE, 4, 256, MIS, FAKE, 64, 32, FAKE, 0, None), 1),     # misaligned codes
    ((FAKE, 4, 256, FAKE, FAKE, 64, 32, None, 0, None), 1),    # null y
    ((None, 0, 256, None, None, 64, 32, None, 0, None), 0),    # m = 0
    ((None, 4, 256, None, None, 0, 32, None, 0, None), 0),     # n = 0
])
def test_linear_fwd_rejects_before_launch(lib, args, status):
    assert lib.tq_linear_fwd(*args) == status


@pytest.mark.parametrize("args,status", [
    ((FAKE, FAKE, 4, 60, 256, FAKE, None, FAKE, 32, FAKE, 0, FAKE, 0, None), 2),  # n % 8
    ((FAKE, FAKE, 4, 64, 256, FAKE, None, FAKE, 32, None, 0, None, 0, None), 1),  # no output
    ((FAKE, None, 4, 64, 256, FAKE, None, FAKE, 32, None, 0, FAKE, 0, None), 1),  # dw needs x
    ((None, FAKE, 4, 64, 256, FAKE, None, FAKE, 32, FAKE, 0, None, 0, None), 1),  # dx needs dy
    ((FAKE, FAKE, 4, 64, 256, FAKE, None, FAKE, 32, FAKE, 3, None, 0, None), 1),  # bad dtype
    ((FAKE, FAKE, 4, 64, 256, None, None, FAKE, 32, FAKE, 0, None, 0, None), 1),  # dx needs codes
    ((FAKE, FAKE, 4, 64, 256, None, MIS, FAKE, 32, FAKE, 0, None, 0, None), 1),   # misaligned codes_t
])
def test_linear_bwd_rejects_before_launch(lib, args, status):
    assert lib.tq_linear_bwd(*args) == status


@pytest.mark.parametrize("args,status", [
    ((FAKE, 64, 200, FAKE, None), 1),   # k % 16
    ((None, 64, 256, FAKE, None), 1),   # null codes
    ((FAKE, 64, 256, MIS, None), 1),    # misaligned output
    ((FAKE, -1, 256, FAKE, None), 1),   # negative
    ((None, 0, 256, None, None), 0),    # empty
])
def test_codes_transpose_rejects_before_launch(lib, args, status):
    assert lib.tq_codes_transpose(*args) == status


def test_batched_rejects_before_launch(lib):
    from paper_2606_18114_gb300.tq import FwdDesc
    arr = (FwdDesc * 2)()
    arr[0] = FwdDesc(FAKE, FAKE, FAKE, FAKE, 64, 256, 32, 0)
    arr[1] = FwdDesc(FAKE, FAKE, FAKE, FAKE, 64, 250, 32, 0)  # k % g
    assert lib.tq_linear_fwd_batched(arr, 2, 1, None) == 1
    assert b"descs[1]" in lib.tq_last_error()
    assert lib.tq_linear_fwd_batched(arr, 1, 17, None) == 1   # m > 16
    assert lib.tq_linear_fwd_batched(arr, 300, 1, None) == 1  # count > max
    assert lib.tq_linear_fwd_batched(None, 0, 1, None) == 0   # nothing to do


def test_quantize_batched_rejects_before_launch(lib):
    from paper_2606_18114_gb300.tq import QuantDesc
    arr = (QuantDesc * 3)()
    arr[0] = QuantDesc(FAKE, FAKE, FAKE, FAKE, 8, 256)
    arr[1] = QuantDesc(FAKE, FAKE, FAKE, FAKE, 8, 96)    # k % g (g = 64)
    arr[2] = QuantDesc(MIS, FAKE, FAKE, FAKE, 8, 256)    # misaligned w
    assert lib.tq_quantize_batched(arr, 2, 64, None) == 1
    assert b"descs[1]" in lib.tq_last_error()
    arr[1] = QuantDesc(None, None, None, None, 0, 256)   # empty entry: skipped
    assert lib.tq_quantize_batched(arr, 3, 64, None) == 1
    assert b"descs[2]" in lib.tq_last_error()
    assert lib.tq_quantize_batched(arr, 1, 48, None) == 1     # bad group size
    assert lib.tq_quantize_batched(arr, 300, 64, None) == 1   # count > max
    assert lib.tq_quantize_batched(arr, -1, 64, None) == 1    # negative count
    assert lib.tq_quantize_batched(None, 2, 64, None) == 1    # null descs
    assert lib.tq_quantize_batched(None, 0, 64, None) == 0    # nothing to do


def test_adamw_requantize_rejects_before_launch(lib):
    """Every argument error is reported before anything touches the device."""
    from paper_2606_18114_gb300.tq import AdamwHparams
    import ctypes
    good = AdamwHparams(2.5e-4, 0.9, 0.95, 1e-8, 0.01, 1.0, 1)
    hp = ctypes.byref(good)
    f = lib.tq_adamw_requantize
    assert f(FAKE, FAKE, FAKE, FAKE, 8, 256, 128, None, FAKE, FAKE, FAKE, None) == 1  # no hparams
    assert b"hparams" in lib.tq_last_error()
    for bad in (AdamwHparams(2.5e-4, 0.9, 0.95, 1e-8, 0.01, 1.0, 0),    # step 0
                AdamwHparams(2.5e-4, 1.0, 0.95, 1e-8, 0.01, 1.0, 1),    # beta1 = 1
                AdamwHparams(2.5e-4, 0.9, -0.1, 1e-8, 0.01, 1.0, 1),    # beta2 < 0
                AdamwHparams(-1e-3, 0.9, 0.95, 1e-8, 0.01, 1.0, 1),     # lr < 0
                AdamwHparams(2.5e-4, 0.9, 0.95, 0.0, 0.01, 1.0, 1),     # eps = 0
                AdamwHparams(2.5e-4, 0.9, 0.95, 1e-8, 0.01, float("nan"), 1)):
        assert f(FAKE, FAKE, FAKE, FAKE, 8, 256, 128, ctypes.byref(bad), FAKE, FAKE, FAKE, None) == 1
    assert f(FAKE, FAKE, FAKE, FAKE, 8, 96, 64, hp, FAKE, FAKE, FAKE, None) == 1     # k % g
    assert f(FAKE, FAKE, FAKE, FAKE, 8, 256, 48, hp, FAKE, FAKE, FAKE, None) == 1    # group size
    assert f(FAKE, MIS, FAKE, FAKE, 8, 256, 128, hp, FAKE, FAKE, FAKE, None) == 1    # misaligned grad
    assert b"grad" in lib.tq_last_error()
    assert f(FAKE, FAKE, None, FAKE, 8, 256, 128, hp, FAKE, FAKE, FAKE, None) == 1   # null m
    assert f(FAKE, FAKE, FAKE, FAKE, 0, 256, 128, hp, FAKE, FAKE, FAKE, None) == 0   # empty: nothing


def test_decoupled_and_alpha_grad_reject_before_launch(lib):
    q, ag = lib.tq_quantize_decoupled, lib.tq_alpha_grad
    assert q(FAKE, 8, 96, 64, None, FAKE, FAKE, FAKE, None) == 1          # k % g
    assert q(FAKE, 8, 256, 48, None, FAKE, FAKE, FAKE, None) == 1         # group size
    assert q(MIS, 8, 256, 128, None, FAKE, FAKE, FAKE, None) == 1         # misaligned w
    assert q(FAKE, 8, 256, 128, FAKE + 2, FAKE, FAKE, FAKE, None) == 1    # misaligned factors
    assert b"row_factor" in lib.tq_last_error()
    assert q(FAKE, 0, 256, 128, None, FAKE, FAKE, FAKE, None) == 0        # empty
    assert ag(FAKE, FAKE, 8, 96, 64, FAKE, None) == 1                     # k % g
    assert ag(FAKE, FAKE, 8, 256, 16, FAKE, None) == 1                    # group size
    assert ag(MIS, FAKE, 8, 256, 128, FAKE, None) == 1                    # misaligned dw
    assert ag(FAKE, FAKE, 8, 256, 128, None, None) == 1                   # null dalpha
    assert ag(FAKE, FAKE, -1, 256, 128, FAKE, None) == 1                  # negative size
    assert ag(FAKE, FAKE, 0, 256, 128, FAKE, None) == 0                   # empty


def test_learnable_scale_entries_reject_before_launch(lib):
    from paper_2606_18114_gb300.tq import AdamwHparams
    import ctypes
    hp = ctypes.byref(AdamwHparams(2.5e-4, 0.9, 0.95, 1e-8, 0.01, 1.0, 1))
    q, sg = lib.tq_quantize_with_scales, lib.tq_scale_grad
    assert q(FAKE, 8, 96, 64, FAKE, FAKE, FAKE, None) == 1                # k % g
    assert q(FAKE, 8, 256, 48, FAKE, FAKE, FAKE, None) == 1               # group size
    assert q(FAKE, 8, 256, 128, None, FAKE, FAKE, None) == 1              # null scales
    assert q(FAKE, 8, 256, 128, MIS, FAKE, FAKE, None) == 1               # misaligned scales
    assert q(FAKE, 0, 256, 128, FAKE, FAKE, FAKE, None) == 0              # empty
    assert sg(FAKE, FAKE, FAKE, FAKE, 8, 96, 64, FAKE, None) == 1         # k % g
    assert sg(FAKE, FAKE, FAKE, FAKE, 8, 256, 16, FAKE, None) == 1        # group size
    assert sg(FAKE, MIS, FAKE, FAKE, 8, 256, 128, FAKE, None) == 1        # misaligned dw
    assert sg(FAKE, FAKE, FAKE, None, 8, 256, 128, FAKE, None) == 1       # null scales
    assert sg(FAKE, FAKE, FAKE, FAKE, 8, 256, 128, None, None) == 1       # null dscales
    assert b"dscales" in lib.tq_last_error()
    assert sg(FAKE, FAKE, FAKE, FAKE, 0, 256, 128, FAKE, None) == 0       # empty
    a = lib.tq_adamw_requantize_with_scales
    assert a(FAKE, FAKE, FAKE, FAKE, 8, 256, 128, None, FAKE, FAKE, FAKE, None) == 1  # no hparams
    assert a(FAKE, FAKE, FAKE, FAKE, 8, 256, 128, hp, None, FAKE, FAKE, None) == 1    # null scales
    assert a(FAKE, FAKE, FAKE, FAKE, 8, 96, 64, hp, FAKE, FAKE, FAKE, None) == 1      # k % g
    assert a(FAKE, FAKE, FAKE, FAKE, 0, 256, 128, hp, FAKE, FAKE, FAKE, None) == 0    # empty
    p = lib.tq_adamw
    assert p(FAKE, FAKE, FAKE, FAKE, 24, hp, None) == 1                   # count % 16
    assert p(FAKE, FAKE, FAKE, FAKE, -16, hp, None) == 1                  # negative count
    assert p(FAKE, FAKE, FAKE, FAKE, 32, None, None) == 1                 # no hparams
    assert p(FAKE, MIS, FAKE, FAKE, 32, hp, None) == 1                    # misaligned grad
    assert p(FAKE, FAKE, FAKE, FAKE, 0, hp, None) == 0                    # empty


def test_activation_flag_checked(lib):
    """The output-type word takes TQ_IN_F16 and nothing else beyond the output type;
    a batched decode takes one activation type."""
    from paper_2606_18114_gb300.tq import FwdDesc
    f = lib.tq_linear_fwd
    assert f(FAKE, 4, 256, FAKE, FAKE, 64, 128, FAKE, 0x200, None) == 1   # unknown flag
    assert f(FAKE, 4, 256, FAKE, FAKE, 64, 128, FAKE, 0x102, None) == 1   # bad output type
    b = lib.tq_linear_bwd
    assert b(FAKE, FAKE, 4, 64, 256, FAKE, None, FAKE, 128, FAKE, 0x400, None, 0, None) == 1
    arr = (FwdDesc * 2)()
    arr[0] = FwdDesc(FAKE, FAKE, FAKE, FAKE, 64, 256, 128, 0)
    arr[1] = FwdDesc(FAKE, FAKE, FAKE, FAKE, 64, 256, 128, 0x100)
    assert lib.tq_linear_fwd_batched(arr, 2, 4, None) == 1
    assert b"activation type" in lib.tq_last_error()


def test_test_hooks_reject_before_device(lib):
    # argument errors come before any device access
    assert lib.tq_test_hooks(-1, 0) == 1
    assert lib.tq_test_hooks(1000, 8) == 1
    assert b"flags" in lib.tq_last_error()
