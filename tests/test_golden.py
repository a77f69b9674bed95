"""The oracle still reproduces its frozen config-1 output (no GPU)."""
import os

import numpy as np

import oracle
from paper_2609_04523_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "cfg1_oracle.txt")


def test_cfg1_golden():
    inp = W.make_config_inputs(1)
    o, lse = oracle.attn_fwd(inp.q, inp.k, inp.v, True, inp.cfg.scale, n_threads=2)
    n_lse = n_o = 0
    with open(GOLDEN) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            parts = line.split()
            h, i = int(parts[1]), int(parts[2])
            vals = np.array([float(x) for x in parts[3:]])
            if parts[0] == "lse":
                assert abs(lse[0, h, i] - vals[0]) <= 1e-12
                n_lse += 1
            else:
                assert np.max(np.abs(o[0, i, h] - vals)) <= 1e-12
                n_o += 1
    assert n_lse == 256 and n_o == 10
