"""Write tests/golden/tiny_attention_seed0.txt from the oracle alone.

The tiny attention configuration (B=1, H=2, Sq=Skv=128, D=64, bf16 Q/K/V i.i.d. N(0,1)
from seed 0, scale = 1/sqrt(64)): the bf16 input checksums, then LSE and four O columns
of six rows per head, non-causal and causal, from oracle.attention (fp64, the attention
definition; the paper prints no worked example, so every stored value is the oracle's).

    python tests/golden/make_golden.py
"""
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
import synth  # noqa: E402

B, H, S, D = 1, 2, 128, 64
ROWS = (0, 1, 2, 63, 64, 127)
COLS = (0, 1, 31, 63)
OUT = os.path.join(HERE, "tiny_attention_seed0.txt")


def inputs():
    return (synth.bf16_normal(0, synth.STREAM_Q, (B, H, S, D)),
            synth.bf16_normal(0, synth.STREAM_K, (B, H, S, D)),
            synth.bf16_normal(0, synth.STREAM_V, (B, H, S, D)))


def checksums(q, k, v):
    return [int(np.asarray(x).astype(np.uint16).astype(np.int64).sum()) for x in (q, k, v)]


def main():
    oracle.build()
    q, k, v = inputs()
    lines = ["# tiny attention B=1 H=2 Sq=Skv=128 D=64 seed 0, scale 1/sqrt(64); written by make_golden.py",
             "# from oracle.attention (fp64 definition).  checksum = sum of the bf16 bit patterns",
             "checksum " + " ".join(str(c) for c in checksums(q, k, v)),
             "# causal head row lse " + " ".join(f"o[{c}]" for c in COLS)]
    for causal in (0, 1):
        o, lse = oracle.attention(q, k, v, causal=bool(causal))
        for h in range(H):
            for r in ROWS:
                vals = [lse[0, h, r]] + [o[0, h, r, c] for c in COLS]
                lines.append(f"{causal} {h} {r} " + " ".join(repr(float(x)) for x in vals))
    with open(OUT, "w") as f:
        f.write("\n".join(lines) + "\n")
    print("wrote", OUT)


if __name__ == "__main__":
    main()
