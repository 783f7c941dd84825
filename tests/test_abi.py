"""The C-ABI library builds, loads without a GPU, exports every entry point that
include/bag.h declares, and rejects bad arguments from its host checks (no device call
is reached for these)."""

import ctypes
import os
import re

import pytest

from paper_2608_09231_gb300 import bag, configs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_09231_gb300 import build
    build.build()
    return bag.load()


def _declared():
    src = open(os.path.join(ROOT, "include", "bag.h")).read()
    return sorted(set(re.findall(r"^\s*(?:bag_status|void|const char\*)\s+(bag_\w+)\(", src, re.M)))


def test_header_declares_the_boundary():
    names = _declared()
    for must in ("bag_create", "bag_step", "bag_run", "bag_reset", "bag_destroy"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name
    assert sorted(bag.EXPORTS) == _declared()


def _create(lib, conf, T, B, tau=0.5, **patch):
    a = bag.arch_from_config(conf, tau)
    for k, v in patch.items():
        setattr(a, k, v)
    h = ctypes.c_void_p()
    st = lib.bag_create(ctypes.byref(a), T, B, ctypes.byref(h))
    return st, h, lib.bag_last_error(None).decode()


@pytest.mark.parametrize("T,B", [(10, 11), (10, 0), (0, 0), (5, -1)])
def test_create_rejects_bad_budget(lib, T, B):
    st, h, msg = _create(lib, configs.get_config("tiny"), T, B)
    assert st == 1 and not h.value and "B" in msg


@pytest.mark.parametrize("patch,code", [
    (dict(heads=3), 1),            # hidden not divisible by heads
    (dict(heads=8), 7),            # head_dim 32 not implemented
    (dict(kind=9), 1),
    (dict(tau=1.0), 1),
    (dict(tau=0.0), 1),
    (dict(patch_ch=16), 7),
    (dict(n_single=0), 1),         # no blocks
    (dict(gate_kind=3), 1),        # unknown gate architecture
    (dict(cfg=2), 1),              # guidance flag is 0 or 1
    (dict(cfg=1, guidance=float("nan")), 1),
    (dict(qk_norm=2), 1),
    (dict(qk_norm=1), 7),          # QK-norm rides on the tensor-core epilogue: bf16 only
    (dict(sampler=2), 1),
    (dict(shift=-1.0), 1),
])
def test_create_rejects_bad_arch(lib, patch, code):
    st, h, msg = _create(lib, configs.get_config("tiny"), 10, 5, **patch)
    assert st == code and not h.value and msg


def test_create_rejects_bad_rope_axes(lib):
    cfg = configs.get_config("tiny")
    a = bag.arch_from_config(cfg)
    a.rope_axes[:] = [0, 30, 32]
    h = ctypes.c_void_p()
    assert lib.bag_create(ctypes.byref(a), 10, 5, ctypes.byref(h)) == 1


def test_null_arguments(lib):
    h = ctypes.c_void_p()
    assert lib.bag_create(None, 10, 5, ctypes.byref(h)) == 1
    assert lib.bag_reset(None) == 1
    assert lib.bag_set_budget(None, 3) == 1
    assert lib.bag_run(None, None, None, None) == 1
    lib.bag_destroy(None)


def test_bf16_backbone_needs_tensor_core_head_dim(lib):
    """bf16 attention runs only on the tensor-core kernel (head_dim 128); a bf16 backbone
    with head_dim 64 is refused at creation instead of running on CUDA cores."""
    a = bag.arch_from_config(configs.get_config("flux_small"))
    a.heads = 8
    a.rope_axes[:] = [16, 24, 24]
    h = ctypes.c_void_p()
    assert lib.bag_create(ctypes.byref(a), 4, 2, ctypes.byref(h)) == 7 and not h.value
    assert "head_dim 128" in lib.bag_last_error(None).decode()


def test_qk_norm_unsupported_for_wan(lib):
    st, h, msg = _create(lib, configs.get_config("wan_small"), 4, 2, qk_norm=1)
    assert st == 7 and not h.value and "qk_norm" in msg
