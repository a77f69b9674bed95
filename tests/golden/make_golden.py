"""Writes tests/golden/cfg1_oracle.txt from the fp64 oracle.

The paper prints no worked example with numbers for its attention kernels
(Table 2 gives only latencies), so no stored value here comes from the paper.
This script freezes what the pinned oracle computes on config 1 (causal MHA,
B=1, Hq=Hkv=2, S=128, D=64, seed 1001), in the spirit of the paper's frozen
test suite (Section 2.4: the tests are written before optimisation and never
changed afterwards).  It calls only oracle/ and the seeded input generator.

Run from the repository root:  python tests/golden/make_golden.py
"""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2609_04523_gb300 import workloads as W  # noqa: E402

ROWS = [0, 1, 63, 64, 127]


def main():
    inp = W.make_config_inputs(1)
    c = inp.cfg
    o, lse = oracle.attn_fwd(inp.q, inp.k, inp.v, c.causal, c.scale)
    out = os.path.join(os.path.dirname(os.path.abspath(__file__)), "cfg1_oracle.txt")
    with open(out, "w") as f:
        f.write("# fp64 oracle on config 1: causal MHA B=1 Hq=Hkv=2 S=128 D=64, seed 1001,\n")
        f.write("# scale 1/8.  Written by tests/golden/make_golden.py (oracle/ only).\n")
        f.write("# lse <h> <i> <value>   |   o <h> <i> <64 values>\n")
        for h in range(c.Hq):
            for i in range(c.S):
                f.write(f"lse {h} {i} {float(lse[0, h, i])!r}\n")
        for h in range(c.Hq):
            for i in ROWS:
                f.write(f"o {h} {i} " + " ".join(repr(float(x)) for x in o[0, i, h]) + "\n")
    print("wrote", out)


if __name__ == "__main__":
    main()
