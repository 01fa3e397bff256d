"""The C-ABI library loads on a host without a GPU and exports exactly the
entry points include/sn.h declares.  No compute calls."""
import os
import re
import subprocess

import pytest

from paper_2110_06037_gb300 import _sn

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            names |= set(re.findall(r"^SN_API[^(]*?\b(sn_\w+)\s*\(", src, flags=re.M))
    return names


def test_header_declares_the_boundary():
    d = _declared()
    for name in ("sn_graph_create", "sn_add_layer", "sn_profile", "sn_select_path", "sn_run"):
        assert name in d


def test_library_exports_every_declared_symbol():
    lib = _sn.lib()
    for name in _declared():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", _sn.LIB_PATH], capture_output=True, text=True).stdout
    exported = set(re.findall(r"\bT (sn_\w+)", out))
    assert _declared() <= exported
    assert exported <= _declared(), f"undeclared exports: {exported - _declared()}"


def test_binding_covers_the_header():
    assert _declared() == set(_sn.SIGNATURES)


def test_routine_names():
    assert _sn.routine_name(1) == "conv2/direct"
    assert _sn.routine_name(999) == "?"
