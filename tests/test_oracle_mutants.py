"""Mutation check of the oracle's pins.

Each case copies oracle.c to a temporary directory, plants one plausible
mistake (a dropped term, a wrong sign or index, a transposed operand), builds
it, and runs every pin in test_oracle_pins.py against it.  A mutant that
passes all the pins would mean the pins cannot see that mistake, so the test
requires each mutant to fail at least one pin.  The real oracle is untouched.
"""
import inspect
import os
import subprocess

import pytest

import oracle
from tests import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

MUTANTS = {
    "scale dropped": ("\n        x[j] = scale * acc;", "\n        x[j] = acc;"),
    "dense scale dropped": ("\n            x[j] = scale * acc;", "\n            x[j] = acc;"),
    "dense head group h%Hkv": ("int g = h / G;\n        double *o = out + (int64_t)h * d;",
                               "int g = h % Hkv;\n        double *o = out + (int64_t)h * d;"),
    "head group h%Hkv": ("ctx_lens[s], max_blocks, h / G, scale, x,", "ctx_lens[s], max_blocks, h % Hkv, scale, x,"),
    "score offset +1": ("        int off = j % bs;\n        double acc = 0.0;",
                        "        int off = (j + 1) % bs;\n        double acc = 0.0;"),
    "V read as K in scores": ("bf16_to_double(pool[kv_elem(blk, page_elems, 0, g, off, c, Hkv, bs, d)]);\n        x[j]",
                              "bf16_to_double(pool[kv_elem(blk, page_elems, 1, g, off, c, Hkv, bs, d)]);\n        x[j]"),
    "softmax sign": ("\n        x[j] = exp(x[j] - m);", "\n        x[j] = exp(m - x[j]);"),
    "denominator dropped": ("double p = x[j] / denom;", "double p = x[j];"),
    "last token skipped": ("    /* weighted sum of values */\n    for (int j = 0; j < n; ++j) {",
                           "    /* weighted sum of values */\n    for (int j = 0; j < n - 1; ++j) {"),
    "append slot n": ("int pos = n - 1;", "int pos = n;"),
    "append K/V swapped": ("pool[kv_elem(blk, page_elems, 0, g, off, c, Hkv, bs, d)] =\n                    k_new",
                           "pool[kv_elem(blk, page_elems, 1, g, off, c, Hkv, bs, d)] =\n                    k_new"),
    "layout head/offset transposed": ("return block * page_elems + (((int64_t)which * Hkv + g) * bs + off) * d + c;",
                                      "return block * page_elems + (((int64_t)which * bs + off) * Hkv + g) * d + c;"),
    "combine weight sign": ("double w = exp(m[i] - M);", "double w = exp(M - m[i]);"),
    "split combine drops the last split": ("for (int i = 0; i < ns; ++i) {\n                double w",
                                           "for (int i = 0; i + 1 < ns; ++i) {\n                double w"),
    "splits overlap by one key": ("int end = start + split_len < n ? start + split_len : n;",
                                  "int end = start + split_len + 1 < n ? start + split_len + 1 : n;"),
    "combine denominator without l": ("denom += w * l[i];", "denom += w;"),
}


def _pin_calls():
    calls = []
    for name, fn in inspect.getmembers(pins, inspect.isfunction):
        if not name.startswith("test_"):
            continue
        marks = getattr(fn, "pytestmark", [])
        params = [m for m in marks if m.name == "parametrize"]
        # every combination of every parametrize mark, as pytest runs them
        combos = [{}]
        for m in params:
            argnames, values = m.args
            argnames = [a.strip() for a in argnames.split(",")]
            combos = [dict(c, **dict(zip(argnames, v if isinstance(v, tuple) else (v,))))
                      for c in combos for v in values]
        for kw in combos:
            calls.append((name, fn, kw))
    out = []
    for name, fn, kw in calls:
        if "oracle_mod" in sig_of(fn):
            kw = dict(kw, oracle_mod=oracle)
        out.append((name, fn, kw))
    return out


def sig_of(fn):
    return inspect.signature(fn).parameters


@pytest.mark.parametrize("mutant", sorted(MUTANTS))
def test_pins_catch_mutant(tmp_path, mutant):
    old, new = MUTANTS[mutant]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor not unique/found: {mutant}"
    path = tmp_path / "oracle_mut.c"
    path.write_text(src.replace(old, new))
    lib = tmp_path / "liboracle_mut.so"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", str(lib), str(path), "-lm"])
    caught = []
    with oracle.swapped_library(str(lib)):
        for name, fn, kw in _pin_calls():
            try:
                fn(**kw)
            except (AssertionError, ValueError):
                caught.append(name)
    assert caught, f"no pin fails on mutant '{mutant}'"
