"""Host-side checks of the C ABI that need no GPU: the library builds, loads
and exports every entry point include/dopr.h declares; the document-side
memory closed form reproduces the paper's printed figures; configuration and
argument validation reject bad input before touching a device."""
import ctypes
import os
import re

import pytest

from paper_2609_03311_gb300 import build as libbuild
from paper_2609_03311_gb300 import dopr, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    libbuild.build()
    return dopr.load()


def header_functions():
    text = open(os.path.join(ROOT, "include", "dopr.h")).read()
    return sorted(set(re.findall(r"DOPR_API[^;(]*?\b(dopr_\w+)\s*\(", text)))


def test_library_exports_every_declared_symbol(lib):
    names = header_functions()
    assert len(names) >= 13
    raw = ctypes.CDLL(dopr.lib_path())
    for n in names:
        assert hasattr(raw, n), f"{n} declared in include/dopr.h but not exported"


def test_version_string(lib):
    assert "sm_103a" in dopr.version()


def test_prefix_bytes_reproduce_paper_memory_tables(lib):
    path = os.path.join(ROOT, "tests", "golden", "paper_doc_memory.csv")
    rows = [l.split(",") for l in open(path) if l.strip() and not l.startswith("#")]
    assert len(rows) >= 20
    for model, tokens, mib, _ in rows:
        cfg = dopr.make_config(synth.MODELS[model])
        got = dopr.prefix_bytes(cfg, int(tokens)) / 2 ** 20
        assert abs(got - float(mib)) < 0.005, (model, tokens, mib, got)


def test_prefix_bytes_compression_ratio_is_eight(lib):
    # Tab. 7: compression ratio 8.0x; e.g. the uncompressed run of a 512-token doc vs m = 64.
    cfg = dopr.make_config(synth.MODELS["qwen3-8b"])
    assert dopr.prefix_bytes(cfg, 512) == 8 * dopr.prefix_bytes(cfg, 64)
    assert dopr.prefix_bytes(cfg, 64) == 64 * 36 * 2 * 8 * 128 * 2


@pytest.mark.parametrize("field,value,status", [
    ("head_dim", 64, dopr.ERR_UNSUPPORTED),
    ("hidden", 1000, dopr.ERR_UNSUPPORTED),
    ("ffn", 100, dopr.ERR_UNSUPPORTED),
    ("n_kv_heads", 3, dopr.ERR_UNSUPPORTED),
    ("n_layers", 0, dopr.ERR_INVALID_ARG),
    ("score_token_id", 151936, dopr.ERR_INVALID_ARG),
    ("max_position", 0, dopr.ERR_INVALID_ARG),
])
def test_bad_config_rejected_before_device_work(lib, field, value, status):
    cfg = dopr.make_config(synth.MODELS["qwen3-0.6b"])
    setattr(cfg, field, value)
    h = ctypes.c_void_p()
    assert lib.dopr_model_create(ctypes.byref(cfg), ctypes.byref(h)) == status
    assert not h.value
    assert lib.dopr_last_error()
    assert lib.dopr_store_create(ctypes.byref(cfg), 10, 1 << 20, ctypes.byref(h)) == status


def test_null_arguments_rejected(lib):
    cfg = dopr.make_config(synth.MODELS["qwen3-0.6b"])
    assert lib.dopr_model_create(None, None) == dopr.ERR_INVALID_ARG
    assert lib.dopr_model_create(ctypes.byref(cfg), None) == dopr.ERR_INVALID_ARG
    assert lib.dopr_store_create(ctypes.byref(cfg), -1, 1 << 20, ctypes.byref(ctypes.c_void_p())) == dopr.ERR_INVALID_ARG
    assert lib.dopr_score(None, None, 1, None, None, None, None, None, 0) == dopr.ERR_INVALID_ARG
    assert lib.dopr_model_destroy(None) == dopr.OK
    assert lib.dopr_store_destroy(None) == dopr.OK
    assert lib.dopr_prefix_bytes(None, 4) == -1
    assert lib.dopr_prefix_bytes(ctypes.byref(cfg), -1) == -1
