"""Writes tests/golden/redraws.json: for each named full-size workload, the
(layer, sequence, original position) rows that near-threshold resampling
redraws, and how often.

The redraws come from the fp64 oracle alone (tests/parity_utils.resample_stack
runs oracle.layer / oracle.keep_top): a token is redrawn while its oracle score
lies within 1e-4 / n of its layer's keep decision (Sec. "Token Pruning", Steps
2-3).  The benchmark and the full-size parity tests draw these workloads with
the stored redraws applied, so the inputs they time and check are the
resampled ones.

    python tests/golden/make_redraws.py            # every workload below
    python tests/golden/make_redraws.py cfg4_L4096_B2_9global
"""
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path[:0] = [ROOT, os.path.join(ROOT, "tests")]

import workloads as wk  # noqa: E402
from parity_utils import resample_stack  # noqa: E402

WORKLOADS = [wk.CFG1, wk.CFG2, wk.CFG3, wk.CFG4] + \
    [wk.cfg5(L) for L in (512, 1024, 2048, 4096)] + [wk.ABS_THETA, wk.TOP_RATIO]
OUT = os.path.join(HERE, "redraws.json")


def main(names):
    try:
        with open(OUT) as f:
            table = json.load(f)
    except FileNotFoundError:
        table = {}
    for wl in WORKLOADS:
        if names and wl.name not in names:
            continue
        _, _, redraws = resample_stack(wl)
        table[wl.name] = {"seed": wl.seed,
                          "redraws": {"%d,%d,%d" % k: c for k, c in sorted(redraws.items())}}
        print(wl.name, len(redraws), "redraws", flush=True)
    with open(OUT, "w") as f:
        json.dump(table, f, indent=1, sort_keys=True)
        f.write("\n")


if __name__ == "__main__":
    main(set(sys.argv[1:]))
