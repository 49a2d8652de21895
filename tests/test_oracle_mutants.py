"""The oracle's pins must catch plausible mistakes.

Each case plants one mistake into a temporary copy of ``oracle/oracle.cpp`` (on the
CPU, in a scratch directory), builds it, swaps it in for the real oracle and checks
that at least one pin of ``test_oracle.py`` fails.
"""
import os
import subprocess

import pytest

import oracle
from tests import test_oracle as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.cpp")

MUTANTS = {
    "dropped_scale": ("const double sj = p.scale * dot;", "const double sj = dot;"),
    "gqa_modulo_map": ("const int hk = h / (p.Hq / p.Hkv);", "const int hk = h % p.Hkv;"),
    "top_left_causal": ("int64_t last = static_cast<int64_t>(i) + (len - p.Sq);",
                        "int64_t last = static_cast<int64_t>(i);"),
    "no_max_subtraction": ("const double w = std::exp(s[static_cast<size_t>(j - j0)] - m);",
                           "const double w = std::exp(s[static_cast<size_t>(j - j0)]); m = 0.0;"),
    "merge_unweighted": ("const double w = std::exp(plse[i] - L);  // exp(-inf) = 0 for empty splits",
                         "const double w = std::isinf(plse[i]) ? 0.0 : 1.0;"),
    "key_stride_transposed": ("return base + ((static_cast<int64_t>(b) * p.Hkv + hk) * p.Skv + j) * p.D;",
                              "return base + ((static_cast<int64_t>(b) * p.Hkv + hk) * p.Skv) * p.D + j;"),
    "lse_without_max": ("return m + std::log(l);", "return std::log(l);"),
}

# pins that take the (swapped) oracle module
PIN_FUNCS = [
    lambda o: pins.test_matches_scipy_softmax(o, 1, 4, 2, 3, 9, 8, True),
    lambda o: pins.test_matches_scipy_softmax(o, 2, 8, 2, 17, 33, 32, False),
    lambda o: pins.test_single_key(o),
    lambda o: pins.test_hard_attention_limit_needs_max_subtraction(o),
    lambda o: pins.test_split_merge_equals_unsplit_for_every_split_count(o, 64),
    lambda o: pins.test_gqa_equals_repeated_kv_heads(o),
    lambda o: pins.test_causal_first_query_sees_only_key0(o),
]


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_mutant(tmp_path, name, monkeypatch):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not found exactly once"
    path = tmp_path / "mutant.cpp"
    path.write_text(src.replace(old, new))
    lib = tmp_path / "libmutant.so"
    subprocess.run(["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-pthread", "-o", str(lib), str(path)],
                   check=True)
    monkeypatch.setattr(oracle, "_lib", oracle._bind(str(lib)))
    caught = 0
    for pin in PIN_FUNCS:
        try:
            pin(oracle)
        except (AssertionError, ValueError, FloatingPointError):
            caught += 1
    assert caught > 0, f"no pin caught mutant {name}"
