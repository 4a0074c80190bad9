"""Writes tests/golden/tiny_oracle.json from the oracle alone.

The paper prints no worked numeric example of the decode step, so the stored
values here are the oracle's own outputs on the seeded tiny workload (2 layers,
hidden 256, vocab 1024, tree 16/4/4, 64 visual + 32 text tokens). They pin the
oracle against accidental change; the oracle itself is pinned by
tests/test_oracle_pins.py. Calls only oracle/ and the input generator.

    python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import msd_oracle as O  # noqa: E402
from paper_2505_14260_gb300 import synth  # noqa: E402
from tests.oracle_support import oracle_model, prompt_numpy  # noqa: E402


def main():
    wl = synth.WORKLOADS["tiny"]
    w = synth.make_weights(wl)
    m = oracle_model(wl, w)
    ids, vis = prompt_numpy(synth.make_prompts(wl)[0])
    st = O.prefill(m, ids, vis)
    steps = []
    for _ in range(wl.steps):
        tree, vr, path, a, bonus = O.spec_step(m, st)
        steps.append({"tokens": tree.tokens.tolist(), "parent": tree.parent.tolist(),
                      "depth": tree.depth.tolist(), "path": path.tolist(),
                      "accept_len": a, "bonus": bonus,
                      "logits_row0_first8": [round(float(x), 9) for x in vr.logits[0, :8]]})
    out = {"workload": "tiny (seed 0, fp32 weights)",
           "weight_checksum": float(sum(float(np.sum(np.abs(v))) for v in
                                        [m.w["embed"], m.w["lm_head"], m.w["draft_fc"]])),
           "prompt_ids": ids.tolist(),
           "greedy_ar": O.greedy_ar(m, ids, vis, len(st.emitted)),
           "spec_emitted": st.emitted,
           "steps": steps}
    with open(os.path.join(os.path.dirname(__file__), "tiny_oracle.json"), "w") as f:
        json.dump(out, f, indent=1)


if __name__ == "__main__":
    main()
