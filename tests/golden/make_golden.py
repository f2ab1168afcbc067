"""Write tests/golden/oracle_tiny.json: the oracle's P(+) and per-layer attention
norms on the seeded tiny workload (2 layers, d=256, 4/2 heads, hd=64, ff=1024,
B=4, L=128), plus a ragged variant.  Calls only oracle/ and kvsynth/.

These values are a cross-machine regression fixture for the oracle (x86 build
host vs Arm GPU host), not a pin: the paper prints no worked numeric example
(Sec. 5 reports only accuracy and latency), so every pin of the oracle's
arithmetic lives in tests/oracle_pins.py."""
import json
import os
import sys

import numpy as np

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))))
import kvsynth as ks  # noqa: E402
import oracle  # noqa: E402


def compute():
    out = {}
    t = ks.Tables.make()
    w = ks.make_workload("tiny")
    r = oracle.score_synth(w, t)
    out["tiny"] = {"p_plus": r.p_plus.tolist(), "attn_absmax": np.abs(r.attn).max(axis=-1).tolist()}
    t2 = ks.Tables.make(0.2)
    w2 = ks.distinct("ragged", ks.ARCH_TINY, 11, [0, 1, 15, 16, 17, 100], gain_std=0.2)
    r2 = oracle.score_synth(w2, t2)
    out["ragged_gain0.2"] = {"p_plus": r2.p_plus.tolist(), "attn_absmax": np.abs(r2.attn).max(axis=-1).tolist()}
    return out


if __name__ == "__main__":
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_tiny.json")
    with open(path, "w") as f:
        json.dump(compute(), f, indent=1)
    print("wrote", path)
