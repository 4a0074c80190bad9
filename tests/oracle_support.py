"""Helpers that hand synthetic workloads to the oracle (tests only)."""
import numpy as np

from oracle.msd_oracle import OracleConfig, OracleModel
from paper_2505_14260_gb300 import synth


def oracle_config(wl: synth.Workload) -> OracleConfig:
    return OracleConfig(n_layers=wl.n_layers, hidden=wl.hidden, n_heads=wl.n_heads,
                        head_dim=wl.head_dim, ffn=wl.ffn, vocab=wl.vocab,
                        tree_nodes=wl.tree_nodes, tree_depth=wl.tree_depth,
                        topk=wl.topk, rms_eps=wl.rms_eps, rope_base=wl.rope_base,
                        draft_input=wl.draft_input)


def oracle_model(wl: synth.Workload, weights_torch: dict) -> OracleModel:
    return OracleModel(oracle_config(wl), synth.weights_to_numpy(weights_torch))


def prompt_numpy(p: synth.Prompt):
    return p.ids.astype(np.int64), synth.to_numpy_f32(p.vis)


def tiny(**kw) -> synth.Workload:
    return synth.WORKLOADS["tiny"].with_(**kw)
