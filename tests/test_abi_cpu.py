"""Host-side checks of the C ABI that need no GPU: the library builds, loads and
exports every function include/mf.h declares, and argument validation rejects
bad problems before any device work."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def mf():
    from paper_2609_02109_gb300 import build
    build.build()
    from paper_2609_02109_gb300 import mf as mod
    return mod


def _declared():
    hdr = open(os.path.join(ROOT, "include", "mf.h")).read()
    hdr = re.sub(r"/\*.*?\*/", "", hdr, flags=re.S)
    return sorted(set(re.findall(r"\b(mf_[a-z_]+)\s*\(", hdr)))


def test_every_declared_function_is_exported(mf):
    names = _declared()
    assert len(names) >= 14
    lib = C.CDLL(mf.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(mf._EXPORTS) == names


def test_status_strings(mf):
    lib = mf.lib()
    assert lib.mf_status_string(0) == b"MF_OK"
    assert lib.mf_status_string(1) == b"MF_EINVAL"
    assert lib.mf_status_string(6) == b"MF_EDEVICE"


def _create(mf, prob, **over):
    keep = {}
    ptr = lambda a: None if a is None else a.ctypes.data  # noqa: E731
    for k in ("n_options", "local_feats", "demand", "weights", "agg_scale", "sla", "obj_w"):
        v = over.get(k, prob.get(k))
        if v is None:
            keep[k] = None
        else:
            keep[k] = np.ascontiguousarray(v, dtype=np.int32 if k == "n_options" else np.float32)
    n = over.get("n_models", int(np.asarray(prob["n_options"]).size))
    p = mf._Problem(n, ptr(keep["n_options"]), over.get("d_local", prob["d_local"]),
                    over.get("hidden1", prob["hidden1"]), over.get("hidden2", prob["hidden2"]),
                    ptr(keep["local_feats"]), ptr(keep["demand"]), ptr(keep["weights"]),
                    ptr(keep["agg_scale"]), ptr(keep["sla"]), ptr(keep["obj_w"]),
                    float(over.get("vram_cap", prob["vram_cap"])), 0.0, over.get("out_act", 0),
                    over.get("objective", 0), over.get("precision", 0), -1)
    h = C.c_void_p()
    st = mf.lib().mf_create(C.byref(p), C.byref(h))
    return st, h


@pytest.mark.parametrize("over", [
    dict(n_models=0), dict(n_models=17), dict(n_options=np.array([12, 0], np.int32)),
    dict(n_options=np.array([12, 256], np.int32)), dict(d_local=0), dict(d_local=29),
    dict(hidden1=0), dict(hidden1=257), dict(hidden2=-1), dict(objective=2), dict(out_act=3),
    dict(precision=7), dict(precision=3), dict(precision=-1), dict(weights=None), dict(sla=None),
    dict(vram_cap=float("nan")),
])
def test_create_rejects_bad_problems(mf, over):
    st, h = _create(mf, W.tiny(), **over)
    assert st == mf.MF_EINVAL and not h.value
    assert mf.lib().mf_last_error()


@pytest.mark.parametrize("precision", [0, 1, 2])  # MF_FP32, MF_BF16, MF_FP32_SIMT
def test_create_accepts_every_precision(mf, precision):
    """Validation passes for the three precisions (without a device the call then fails
    in the CUDA runtime, not in validation)."""
    st, h = _create(mf, W.paper_scale(), precision=precision)
    assert st != mf.MF_EINVAL, mf.lib().mf_last_error()
    if st == mf.MF_OK:
        mf.lib().mf_destroy(h)
    assert mf.MF_FP32_SIMT == 2 and mf._PRECISIONS["fp32_simt"] == mf.MF_FP32_SIMT


def test_create_rejects_space_overflow(mf):
    prob = W.make_problem([255] * 9, 8, 32, 0, 1, 100.0)
    st, _ = _create(mf, prob)
    assert st == mf.MF_EINVAL
    assert b"overflow" in mf.lib().mf_last_error()


def test_null_arguments(mf):
    lib = mf.lib()
    assert lib.mf_create(None, None) == mf.MF_EINVAL
    assert lib.mf_destroy(None) == mf.MF_OK
    assert lib.mf_space_size(None, None) == mf.MF_EINVAL
    assert lib.mf_search_exhaustive(None, 4, 0, None, None) == mf.MF_EINVAL
    assert lib.mf_ga_generation(None, None, 4, None, None) == mf.MF_EINVAL
