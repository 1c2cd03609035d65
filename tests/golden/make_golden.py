"""Writes oracle_tiny.json: values of the fp64 oracle on small seeded inputs.

The paper prints no worked numeric example, so the stored values here are the
oracle's own, written by this script (which calls only `oracle/` and the
seeded input generator). tests/test_golden.py checks that the oracle still
reproduces them; regenerate only with a change to the oracle's arithmetic,
and name in the commit the passage of the paper that justifies the change.

    python tests/golden/make_golden.py
"""

import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
from paper_2608_08878_gb300 import synth  # noqa: E402


def golden():
    wl = synth.TINY.with_(steps=4)
    blob = synth.policy_weights(wl.policy_seed, wl.mlp_hidden)
    out = {"workload": wl.name, "rows": {}}
    for r in range(wl.rows):
        layer, b, g = wl.row_coords(r)
        row = oracle.OracleRow(wl.head_dim, wl.group, wl.window, wl.alpha_mode, wl.capacity)
        k, v = synth.prompt_row(wl, layer, b, g)
        row.append(k, v)
        steps = []
        for s in range(wl.steps):
            q, kn, vn = synth.step_row(wl, s, layer, b, g)
            res = row.step(q, kn, vn, blob, wl.mlp_hidden, wl.layernorm)
            row.evict(wl.budget)
            steps.append({"o_row0": res["o"][0, :8].tolist(), "Hq": res["Hq"].tolist(),
                          "feat_first4": res["feat"][:4].tolist(), "score_first8": res["score"][:8].tolist(),
                          "kept_positions": row.positions().tolist()})
        out["rows"][str(r)] = steps
    rng = np.random.default_rng(2026)
    s = rng.standard_normal(40) * 2.0
    out["pl_logz"] = [{"B": B, "tau": tau, "logz": oracle.pl_logz(s, B, tau)} for B, tau in ((1, 1.0), (7, 1.0), (40, 0.5))]
    out["pl_scores"] = s.tolist()
    g = rng.gumbel(size=40).astype(np.float32)
    out["gumbel"] = g.tolist()
    out["gumbel_top7"] = oracle.gumbel_topb(s.astype(np.float32), g, 7, 1.0).tolist()
    return out


if __name__ == "__main__":
    oracle.build()
    with open(os.path.join(HERE, "oracle_tiny.json"), "w") as f:
        json.dump(golden(), f, indent=1)
    print("wrote", os.path.join(HERE, "oracle_tiny.json"))
