"""C-ABI checks that need no GPU: the library builds, loads, exports every entry
point declared in include/hero.h, and rejects invalid arguments on the host
before any CUDA call."""

import ctypes
import os
import re

import numpy as np
import pytest

from paper_2609_08189_gb300 import build
from synth import hero_inputs as hi

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def H():
    build.build()
    from paper_2609_08189_gb300 import hero
    hero.load()
    return hero


def declared_functions():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"^\s*(?:[\w\*]+\s+)+\**(hero_\w+)\s*\(", src, flags=re.M))
    return sorted(names)


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("hero_init_weights", "hero_routed_ffn_stack", "hero_free", "hero_last_error"):
        assert n in names


def test_binding_flags_match_the_header(H):
    """The binding's HERO_FLAG_* constants are the header's enum values."""
    src = open(os.path.join(ROOT, "include", "hero.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    flags = {n: int(v) for n, v in re.findall(r"(HERO_FLAG_\w+)\s*=\s*(\d+)u", src)}
    assert set(flags) == {"HERO_FLAG_DENSE", "HERO_FLAG_FORCE_MASK", "HERO_FLAG_HOST_IO",
                          "HERO_FLAG_NO_SPECULATE"}
    for n, v in flags.items():
        assert getattr(H, n) == v, n
    assert len(set(flags.values())) == len(flags) and all(v & (v - 1) == 0 for v in flags.values())


def test_library_exports_every_declared_symbol(H):
    lib = ctypes.CDLL(H.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_init_rejects_bad_configs_on_host(H):
    w = hi.generate_weights(hi.CONFIGS["tiny_f32"])
    out = ctypes.c_void_p()
    lib = H.load()
    # NULL config / NULL weights / NULL out
    assert lib.hero_init_weights(None, None, ctypes.byref(out)) == H.HERO_ERR_ARG
    assert "NULL" in H.hero_last_error()
    cfg = H.make_config(hi.CONFIGS["tiny_f32"])
    assert lib.hero_init_weights(ctypes.byref(cfg), None, ctypes.byref(out)) == H.HERO_ERR_ARG
    ws, keep = H.make_weights(w)
    assert lib.hero_init_weights(ctypes.byref(cfg), ctypes.byref(ws), None) == H.HERO_ERR_ARG
    # unsupported memory width and bad dimensions
    for bad, code in [(dict(d_m=24), H.HERO_ERR_UNSUPPORTED), (dict(n_layers=0), H.HERO_ERR_ARG),
                      (dict(d_enc=300), H.HERO_ERR_UNSUPPORTED), (dict(d_model=250), H.HERO_ERR_UNSUPPORTED)]:
        c = H.make_config(hi.CONFIGS["tiny_f32"].replace(**bad))
        assert lib.hero_init_weights(ctypes.byref(c), ctypes.byref(ws), ctypes.byref(out)) == code, bad
        assert out.value is None
    # bf16 shape rules
    c = H.make_config(hi.CONFIGS["small_bf16"].replace(d_ff=1000))
    assert lib.hero_init_weights(ctypes.byref(c), ctypes.byref(ws), ctypes.byref(out)) == H.HERO_ERR_UNSUPPORTED
    # a NULL parameter pointer
    ws2 = H.hero_weights_host(ws.host_dtype, *[getattr(ws, n) for n in H.WEIGHT_FIELDS])
    ws2.w_k = None
    assert lib.hero_init_weights(ctypes.byref(cfg), ctypes.byref(ws2), ctypes.byref(out)) == H.HERO_ERR_ARG
    # bf16 host arrays for an f32 model
    wb = hi.generate_weights(hi.CONFIGS["small_bf16"])
    wsb, keepb = H.make_weights(wb)
    assert lib.hero_init_weights(ctypes.byref(cfg), ctypes.byref(wsb), ctypes.byref(out)) == H.HERO_ERR_ARG
    del keep, keepb


def test_stack_rejects_null_model(H):
    lib = H.load()
    assert lib.hero_routed_ffn_stack(None, 1, None, None, 0.5, 0, None, None, None, None, None,
                                     None) == H.HERO_ERR_ARG
    assert lib.hero_check_device_status(None, None) == H.HERO_ERR_ARG
    assert lib.hero_set_profiling(None, 1) == H.HERO_ERR_ARG
    lib.hero_free(None)  # NULL-safe


def test_binding_fails_loudly_without_library(tmp_path, monkeypatch):
    from paper_2609_08189_gb300 import hero
    monkeypatch.setattr(hero, "_lib", None)
    with pytest.raises(RuntimeError):
        hero.load(str(tmp_path / "missing.so"))
