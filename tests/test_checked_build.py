"""The checked build (host only, no GPU): compiled with -DDOPR_CHECKED it tests
every data-dependent global index against its buffer (a memory checker's job,
with no tool that can fault the GPU).  Here: it builds, exports every entry
point the header declares, and the status it reports a skipped access with is
declared in the header and named by the binding."""
import ctypes
import os
import re

from paper_2609_03311_gb300 import build as libbuild
from paper_2609_03311_gb300 import dopr

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_checked_library_builds_and_exports_every_declared_symbol():
    path = libbuild.build(checked=True)
    assert path == libbuild.LIB_CHECKED and path != libbuild.LIB
    text = open(os.path.join(ROOT, "include", "dopr.h")).read()
    names = sorted(set(re.findall(r"DOPR_API[^;(]*?\b(dopr_\w+)\s*\(", text)))
    raw = ctypes.CDLL(path)
    for n in names:
        assert hasattr(raw, n), f"{n} missing from the checked build"
    raw.dopr_version.restype = ctypes.c_char_p
    assert b"sm_103a" in raw.dopr_version()


def test_internal_status_declared_and_named():
    text = open(os.path.join(ROOT, "include", "dopr.h")).read()
    assert re.search(r"DOPR_ERR_INTERNAL\s*=\s*8\b", text)
    assert dopr.ERR_INTERNAL == 8 and dopr.STATUS_NAMES[8] == "INTERNAL"


def test_binding_selects_the_checked_library(monkeypatch):
    monkeypatch.setenv("DOPR_CHECKED", "1")
    assert dopr.lib_path() == libbuild.LIB_CHECKED
    monkeypatch.delenv("DOPR_CHECKED")
    assert dopr.lib_path() == libbuild.LIB
