"""The oracle reproduces its stored outputs on the seeded tiny workload
(written by tests/golden/make_golden.py, which calls only the oracle)."""
import json
import os

import numpy as np
import pytest

from oracle import msd_oracle as O
from paper_2505_14260_gb300 import synth
from tests.oracle_support import oracle_model, prompt_numpy

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "tiny_oracle.json")


def test_oracle_matches_golden_tiny():
    d = json.load(open(GOLDEN))
    wl = synth.WORKLOADS["tiny"]
    m = oracle_model(wl, synth.make_weights(wl))
    csum = float(sum(float(np.sum(np.abs(v))) for v in
                     [m.w["embed"], m.w["lm_head"], m.w["draft_fc"]]))
    if abs(csum - d["weight_checksum"]) > 1e-6 * abs(csum):
        pytest.skip("this torch build draws different CPU random numbers")
    ids, vis = prompt_numpy(synth.make_prompts(wl)[0])
    assert ids.tolist() == d["prompt_ids"]
    st = O.prefill(m, ids, vis)
    for s in d["steps"]:
        tree, vr, path, a, bonus = O.spec_step(m, st)
        assert tree.tokens.tolist() == s["tokens"] and tree.parent.tolist() == s["parent"]
        assert path.tolist() == s["path"] and a == s["accept_len"] and bonus == s["bonus"]
        np.testing.assert_allclose(vr.logits[0, :8], s["logits_row0_first8"], atol=2e-9)
    assert st.emitted == d["spec_emitted"] == d["greedy_ar"]
