"""Stored oracle values for the tiny attention configuration (tests/golden/, written by
tests/golden/make_golden.py from the oracle alone).  On every machine the seeded bf16
inputs must reproduce the stored bit checksums and the oracle the stored values, so that
the generator and the oracle behave identically on the x86 host and the Arm GPU hosts."""
import os
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.join(HERE, "golden"))

import make_golden  # noqa: E402
import oracle  # noqa: E402


def load():
    checks, rows = None, []
    with open(os.path.join(HERE, "golden", "tiny_attention_seed0.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            parts = line.split()
            if parts[0] == "checksum":
                checks = [int(x) for x in parts[1:]]
            else:
                rows.append((int(parts[0]), int(parts[1]), int(parts[2]), [float(x) for x in parts[3:]]))
    return checks, rows


def test_generator_reproduces_stored_bits():
    checks, _ = load()
    assert make_golden.checksums(*make_golden.inputs()) == checks


def test_oracle_reproduces_stored_values():
    _, rows = load()
    q, k, v = make_golden.inputs()
    outs = {c: oracle.attention(q, k, v, causal=bool(c)) for c in (0, 1)}
    for causal, h, r, vals in rows:
        o, lse = outs[causal]
        got = [lse[0, h, r]] + [o[0, h, r, c] for c in make_golden.COLS]
        np.testing.assert_allclose(got, vals, rtol=1e-12, atol=1e-14)


def test_causal_row_zero_is_v0():
    # a closed form inside the stored data: the first causal query attends to key 0 only
    import synth
    _, rows = load()
    _, _, v = make_golden.inputs()
    vf = synth.bf16_to_f32(v).astype(np.float64)
    zero_rows = [(h, vals) for causal, h, r, vals in rows if causal == 1 and r == 0]
    assert zero_rows
    for h, vals in zero_rows:
        np.testing.assert_allclose(vals[1:], [vf[0, h, 0, c] for c in make_golden.COLS], rtol=0, atol=1e-12)
