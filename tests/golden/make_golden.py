"""Writes the stored oracle fixtures in this folder.  Calls only ``oracle``
(and the seeded input generator); run from the repository root:

    python tests/golden/make_golden.py
"""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
from paper_2412_15803_gb300 import synth  # noqa: E402

CASES = [  # (seed, N, K, batch)
    (0, 8, 256, 1),
    (5, 6, 288, 2),
]


def main():
    path = os.path.join(HERE, "gemv_small.txt")
    with open(path, "w") as f:
        f.write("# oracle GEMV fixtures: seed N K batch, then y16 bits [batch][N] in hex\n")
        f.write("# inputs: paper_2412_15803_gb300.synth.matrix(seed, N, K) and activations(seed, batch, K)\n")
        for seed, N, K, batch in CASES:
            W, s = synth.matrix(seed, N, K)
            x = synth.activations(seed, batch, K)
            _, _, y16 = oracle.gemv(W, s, x)
            f.write(f"case {seed} {N} {K} {batch}\n")
            for b in range(batch):
                f.write(" ".join(f"{int(v):04x}" for v in y16[b]) + "\n")
    print("wrote", path)


if __name__ == "__main__":
    main()
