"""The C-ABI library loads and exports every function include/rheo.h declares;
host-side validation rejects bad configurations without touching a GPU."""
import ctypes
import os
import re

import pytest

from paper_2609_21827_gb300 import build, rheo, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return rheo.lib()


def declared():
    src = open(os.path.join(ROOT, "include", "rheo.h")).read()
    return sorted(set(re.findall(r"^int\s+(rheo_\w+)\s*\(", src, flags=re.M)))


def test_header_declares_the_entry_points():
    assert declared() == sorted(rheo.EXPORTS)


def test_every_declared_symbol_is_exported(lib):
    for name in declared():
        assert hasattr(lib, name), name
    raw = ctypes.CDLL(rheo.library_path())
    for name in declared():
        assert ctypes.cast(getattr(raw, name), ctypes.c_void_p).value


@pytest.mark.parametrize("name", list(synth.WORKLOADS))
def test_sizes_of_the_workloads(lib, name):
    w = synth.WORKLOADS[name]
    cfg = rheo.Config(batch=w.batch, vocab=w.vocab, K=w.K, depth=w.depth, budget=w.budget, m=w.m, dtype=w.dtype)
    G1, E, ws = cfg.sizes()
    assert G1 == 1 + (w.K + 1) + (w.depth - 1) * w.K * (w.K + 1)
    assert E == 1 + (w.depth - 1) * w.K
    assert 0 < ws < 2**31


@pytest.mark.parametrize("bad", [dict(m=5, K=4), dict(support=4, K=4), dict(budget=0), dict(budget=10**6),
                                 dict(K=0, depth=2), dict(m=0, eps=0.0), dict(vocab=300000), dict(vocab=262145),
                                 dict(dtype="f16"),
                                 dict(K=127, depth=3), dict(batch=70000), dict(batch=0), dict(vocab=0),
                                 dict(depth=0), dict(K=-1), dict(m=-1), dict(support=129, K=4)])
def test_invalid_configurations_are_rejected(lib, bad):
    # (the largest vocabulary accepted is 262,144; tests/test_gpu_parity.py runs it)
    base = dict(batch=2, vocab=1000, K=4, depth=3, budget=10, m=1)
    base.update(bad)
    cfg = rheo.Config(**base)
    if cfg.dtype not in ("bf16", "f32"):
        c = cfg.c()
        c.dtype = 7
        assert lib.rheo_sizes(ctypes.byref(c), None, None, None) == rheo.RHEO_EINVAL
        return
    with pytest.raises(rheo.RheoError):
        cfg.sizes()


def test_null_pointers_rejected_on_the_host(lib):
    cfg = rheo.Config(batch=2, vocab=1000, K=4, depth=3, budget=10)
    t = rheo._Tree()
    rc = lib.rheo_expand(ctypes.byref(cfg.c()), 1, None, 1000, None, None, None, ctypes.byref(t), None, None)
    assert rc == rheo.RHEO_EINVAL
    rc = lib.rheo_prune(ctypes.byref(cfg.c()), ctypes.byref(t), ctypes.byref(rheo._Pruned()), None, None)
    assert rc == rheo.RHEO_EINVAL
