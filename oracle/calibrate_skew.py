"""Fit the per-expert logit offsets that give the video / stress layers their
skewed expert loads, and store them in ``workloads/skew_offsets.json``.

Test infrastructure: it calls only the oracle (fp64 logits and selection) and
the seeded generator.  It runs once, offline; the generator then reads the
stored offsets as plain input data.

Method: with the constant feature ``x[:, d-1] = 1`` every logit of expert e is
``s0[t, e] + o_e`` where ``s0`` are the logits of the unskewed layer.  Starting
from ``o = 0``, the damped fixed-point step ``o_e += clip(eta * (log(target_e + 1)
- log(count_e + 1)), +-0.5)``, with ``o_e <= 10``, moves each expert's realised
load towards its target (larger steps saturate several sigmoids at once, after
which the bias alone orders those experts and the iteration stalls); empty
experts are pinned at ``o_e = -40`` (sigmoid ~ 4e-18, so the bias alone, at most
0.1, cannot lift them into any top-k).  Offsets are rounded to fp32 (the dtype of
W_r) and the realised loads are re-measured on the final layer.

Usage: ``python oracle/calibrate_skew.py [c3 c4]``
"""
from __future__ import annotations

import json
import os
import sys
import time

import numpy as np

_ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, _ROOT)

import oracle  # noqa: E402
import workloads  # noqa: E402


def fit(name: str, iters: int = 200, eta: float = 0.3):
    cfg = workloads.CONFIGS[name]
    lay = workloads.skew_layout(cfg)
    target, empty = lay["target"], lay["empty"]
    E, T, k = cfg.E, cfg.T, cfg.k
    base = workloads.make_layer(cfg, skew_offsets=np.zeros(E, np.float32))
    t0 = time.time()
    s0 = oracle.logits(base.x, base.Wr)
    print(f"[{name}] base logits in {time.time() - t0:.1f}s", flush=True)
    o = np.zeros(E, np.float64)
    o[empty] = -40.0
    best = None
    for it in range(iters):
        idx, _, _ = oracle.select(s0 + o[None, :], base.b, k)
        counts = np.bincount(idx.ravel(), minlength=E).astype(np.float64)
        err = np.abs(np.log(counts + 1) - np.log(target + 1))
        err[empty] = 0.0
        score = err.max()
        if best is None or score < best[0]:
            best = (score, o.copy(), counts.copy())
        if it % 10 == 0:
            print(f"[{name}] it {it:3d} max|log err| {score:.4f}", flush=True)
        step = eta * (np.log(target + 1) - np.log(counts + 1))
        step[empty] = 0.0
        o = np.minimum(o + np.clip(step, -0.5, 0.5), 10.0)
        o[empty] = -40.0
    o = best[1].astype(np.float32)
    # re-measure on the real layer (offsets applied through W_r[d-1, :])
    lay_final = workloads.make_layer(cfg, skew_offsets=o)
    idx, _, margin = oracle.route(lay_final.x, lay_final.Wr, lay_final.b, k)
    counts = np.bincount(idx.ravel(), minlength=E)
    print(f"[{name}] realised: max {counts.max()} min-nonempty {counts[counts > 0].min()} "
          f"zeros {int((counts == 0).sum())} (target zeros {empty.size}); min margin {margin.min():.3e}")
    return {
        "offsets": [float(v) for v in o],
        "target": [float(v) for v in target],
        "realised_counts": [int(v) for v in counts],
        "empty_experts": [int(v) for v in empty],
        "hot_experts": [int(v) for v in lay["hot"]],
        "min_margin": float(margin.min()),
        "note": "W_r[d-1, e] = offsets[e] with x[:, d-1] = 1; fitted by oracle/calibrate_skew.py",
    }


def main(argv):
    names = argv[1:] or ["c3", "c4"]
    table = {}
    if os.path.exists(workloads.SKEW_FILE):
        with open(workloads.SKEW_FILE) as f:
            table = json.load(f)
    for name in names:
        table[name] = fit(name)
        with open(workloads.SKEW_FILE, "w") as f:
            json.dump(table, f, indent=1)
            f.write("\n")
    print("wrote", workloads.SKEW_FILE)


if __name__ == "__main__":
    main(sys.argv)
