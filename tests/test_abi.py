"""The C-ABI library builds, loads and exports every symbol include/ravel.h
declares; host-side argument checks answer without touching a GPU."""
import ctypes as C
import os
import re

import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_34170_gb300 import build, load
    build.build()
    return load()


def _declared():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(ravel_\w+)\s*\(", src))
    return names


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert {"ravel_create", "ravel_reset", "ravel_set_context", "ravel_roll_step", "ravel_destroy"} <= names
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings(lib):
    from paper_2609_34170_gb300 import ravel_status_string
    assert ravel_status_string(0) == "ok"
    assert "pending" in ravel_status_string(6)
    assert ravel_status_string(99) == "unknown status"


def test_create_rejects_bad_shapes_without_a_gpu(lib):
    from paper_2609_34170_gb300 import RavelError, ravel_create
    cfg = synth.PRESETS["tiny_fp32_b1"]
    W = synth.make_weights(cfg)
    for bad in (cfg.replace(n_q_heads=3, n_kv_heads=2), cfg.replace(head_dim=12), cfg.replace(mlp_dim=100),
                cfg.replace(width=3), cfg.replace(layers=0)):
        with pytest.raises(RavelError) as ei:
            ravel_create(bad, synth.make_weights(bad) if bad.layers else W)
        assert ei.value.status == 2
    # null handles / arguments are refused
    assert lib.ravel_roll_step(None, None, None, None, None, None, None, None) == 1
    assert lib.ravel_set_context(None, None, None, 1, None) == 1
    assert lib.ravel_create(None, None, 0, None) == 1
    lib.ravel_destroy(None)
