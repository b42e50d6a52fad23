"""The C-ABI library loads and exports every entry point include/pad.h declares."""
import os
import re
import subprocess

from paper_2607_02963_gb300 import binding

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "pad.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"\b(pad_[a-z0-9_]+)\s*\(", src)
    return sorted(set(names))


def test_header_declares_the_three_step_calls():
    names = declared_functions()
    for n in ("pad_plan", "pad_kv_append", "pad_event_decode_attn"):
        assert n in names


def test_every_declared_symbol_is_exported(padlib):
    out = subprocess.run(["nm", "-D", "--defined-only", binding.lib_path()], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (pad_[a-z0-9_]+)$", out, flags=re.M))
    missing = [n for n in declared_functions() if n not in exported]
    assert not missing, f"declared but not exported: {missing}"
    for n in declared_functions():
        assert hasattr(padlib, n)


def test_binding_covers_every_declared_symbol():
    assert sorted(binding._SIGNATURES) == declared_functions()


def test_status_strings(padlib):
    for code, name in binding.STATUS_NAMES.items():
        assert padlib.pad_status_string(code).decode() == name
