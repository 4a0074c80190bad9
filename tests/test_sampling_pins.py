"""Pins of the oracle's speculative sampling at temperature T > 0 (Sec. 3.2,
Eq. 6 and the adjusted distribution after it; reading R7 of the oracle).

Against closed forms on a hand-built four-token case, against the defining
property of speculative sampling -- the emitted tokens are distributed exactly
as sampling the target -- by chi-square tests on the tiny model's own verify
distributions, and against greedy acceptance in the zero-temperature limit.
"""
import numpy as np
import pytest
from scipy import stats

from oracle import msd_oracle as O
from paper_2505_14260_gb300 import synth
from tests.oracle_support import oracle_model, prompt_numpy, tiny


def _tree(tokens, parent):
    depth = [0] * len(tokens)
    for i in range(1, len(tokens)):
        depth[i] = depth[parent[i]] + 1
    return O.Tree(tokens=np.array(tokens), parent=np.array(parent), depth=np.array(depth))


P = np.array([0.1, 0.2, 0.3, 0.4])
ROWS = np.log(np.array([P, [0.25] * 4, [0.2, 0.2, 0.2, 0.4], [0.7, 0.1, 0.1, 0.1]]))
TREE = _tree([9, 3, 2, 0], [-1, 0, 0, 1])     # root; children 3 and 2; token 0 under 3
K = 2


def _u(rows):
    u = np.full((3, K + 1), 0.999)
    for (d, j), v in rows.items():
        u[d, j] = v
    return u


def test_sample_index_inverse_cdf():
    assert O.sample_index(P, 0.0) == 0
    assert O.sample_index(P, 0.09) == 0
    assert O.sample_index(P, 0.11) == 1
    assert O.sample_index(P, 0.61) == 3
    assert O.sample_index(P, 0.5, removed=[3, 2]) == 1      # (0.1, 0.2) renormalised: 0.5 * 0.3 = 0.15
    assert O.sample_index(P, 0.3, removed=[3, 2]) == 0      # 0.09 < 0.1
    assert O.sample_index(P, 0.999, removed=[0]) == 3


def test_accept_sample_handbuilt_cases():
    # x = 3 accepted (u < p = 0.4); at node 1 the child token 0 accepted (0.2 < 0.25);
    # node 3 is a leaf: the token is drawn from its own p (cumsum 0.7, 0.8 > 0.75 -> 1)
    path, a, bonus = O.accept_sample(TREE, ROWS, 1.0, _u({(0, 0): 0.39, (1, 0): 0.2, (2, K): 0.75}), K)
    assert list(path) == [0, 1, 3] and a == 2 and bonus == 1
    # 3 rejected (0.41 >= 0.4); 2 tried against p with 3 removed: 0.6 * 0.6 = 0.36 >= 0.3,
    # rejected; the token is drawn from (0.1, 0.2) renormalised: 0.5 * 0.3 = 0.15 -> 1
    path, a, bonus = O.accept_sample(TREE, ROWS, 1.0, _u({(0, 0): 0.41, (0, 1): 0.6, (0, K): 0.5}), K)
    assert list(path) == [0] and a == 0 and bonus == 1
    # 3 rejected, 2 accepted (0.49 * 0.6 = 0.294 < 0.3); node 2 is a leaf: drawn from
    # its p (cumsum 0.2, 0.4, 0.6 > 0.55 -> 2)
    path, a, bonus = O.accept_sample(TREE, ROWS, 1.0, _u({(0, 0): 0.41, (0, 1): 0.49, (1, K): 0.55}), K)
    assert list(path) == [0, 2] and a == 1 and bonus == 2
    # temperature: p ~ exp(log P / T); at T = 0.5, p(3) = 0.16 / 0.30 = 0.533
    pt = P ** 2 / np.sum(P ** 2)
    path, a, _ = O.accept_sample(TREE, ROWS, 0.5, _u({(0, 0): pt[3] - 1e-6}), K)
    assert a >= 1 and path[1] == 1
    path, a, _ = O.accept_sample(TREE, ROWS, 0.5, _u({(0, 0): pt[3] + 1e-6, (0, 1): 0.999}), K)
    assert a == 0


@pytest.fixture(scope="module")
def drafted():
    wl = tiny(n_layers=2)
    w = synth.make_weights(wl)
    m = oracle_model(wl, w)
    ids, vis = prompt_numpy(synth.make_prompts(wl)[0])
    st = O.prefill(m, ids, vis)
    tree = O.draft_tree(m, st)
    vr = O.verify(m, st, tree)
    return wl, tree, vr, m, st


def _chi2_p(counts, probs):
    """Chi-square p-value of counts against probabilities, merging the
    categories expected fewer than 5 times into one."""
    n = counts.sum()
    e = probs * n
    big = e >= 5
    obs = np.append(counts[big], counts[~big].sum())
    exp = np.append(e[big], e[~big].sum())
    if exp[-1] < 5:
        obs, exp = obs[:-1], exp[:-1]
    exp = exp * obs.sum() / exp.sum()
    return stats.chisquare(obs, exp).pvalue


@pytest.mark.parametrize("temperature", [0.1, 1.0])
def test_first_token_is_distributed_as_target_sampling(drafted, temperature):
    wl, tree, vr, _, _ = drafted
    k = wl.topk
    rng = np.random.default_rng(7)
    n = 6000
    first = np.zeros(wl.vocab, np.int64)
    for _ in range(n):
        path, a, bonus = O.accept_sample(tree, vr.logits, temperature, rng.random((wl.tree_depth + 1, k + 1)), k)
        first[int(tree.tokens[path[1]]) if a >= 1 else bonus] += 1
    p_root = O.softmax(np.asarray(vr.logits[0], np.float64) / temperature)
    assert _chi2_p(first, p_root) > 1e-3


def test_second_token_given_an_accepted_child_is_target_sampling(drafted):
    """Given that the root's child c was accepted, the next token is distributed
    as the target at c (the walk continues there, or draws from it). The tree
    is planted so that children are accepted often: the root's children are the
    target's k likeliest tokens (the root's row sees only the prefix, so its
    distribution does not depend on them), and the likeliest child gets k
    children of its own."""
    wl, tree0, vr0, m, st = drafted
    k, T = wl.topk, 0.1
    p_root = O.softmax(np.asarray(vr0.logits[0], np.float64) / T)
    top = O.topk_ids(p_root, k)
    toks = [int(tree0.tokens[0])] + [int(x) for x in top] + [int(x) for x in tree0.tokens[1:k + 1]]
    parent = [-1] + [0] * k + [1] * k
    tree = _tree(toks, parent)
    vr = O.verify(m, st, tree)
    np.testing.assert_allclose(vr.logits[0], vr0.logits[0], rtol=0, atol=1e-12)
    rng = np.random.default_rng(11)
    second = np.zeros(wl.vocab, np.int64)
    for _ in range(6000):
        path, a, bonus = O.accept_sample(tree, vr.logits, T, rng.random((wl.tree_depth + 1, k + 1)), k)
        if a >= 1 and path[1] == 1:
            second[int(tree.tokens[path[2]]) if a >= 2 else bonus] += 1
    assert second.sum() > 200
    assert _chi2_p(second, O.softmax(np.asarray(vr.logits[1], np.float64) / T)) > 1e-3


def test_zero_temperature_limit_is_greedy_acceptance(drafted):
    wl, tree, vr, _, _ = drafted
    rng = np.random.default_rng(3)
    path_g, a_g, bonus_g = O.accept(tree, vr.argmax)
    for _ in range(20):
        path, a, bonus = O.accept_sample(tree, vr.logits, 1e-4, rng.random((wl.tree_depth + 1, wl.topk + 1)),
                                         wl.topk)
        assert list(path) == list(path_g) and a == a_g and bonus == bonus_g


def test_duplicate_sibling_tokens_add_no_mass():
    """A caller-planted tree may repeat a token among siblings: once rejected,
    the token has no mass left in the adjusted distribution, so its duplicate
    is never accepted and the draw excludes it (the emitted distribution is
    that of the tree without the duplicate)."""
    tree = _tree([9, 3, 3, 2], [-1, 0, 0, 0])
    rows = np.repeat(ROWS[:1], 4, axis=0)      # every node's row: the root's p (only the root is visited)
    u = np.full((2, 4), 0.999)
    u[0, 0] = 0.41                       # 3 rejected (0.41 >= 0.4)
    u[0, 1] = 0.0                        # the duplicate 3: p_adj(3) = 0, rejected even at u = 0
    u[0, 2] = 0.99                       # 2 rejected: 0.99 * 0.6 >= 0.3
    u[0, 3] = 0.5                        # draw from (0.1, 0.2) renormalised: 0.5 * 0.3 = 0.15 -> 1
    path, a, bonus = O.accept_sample(tree, rows, 1.0, u, 3)
    assert list(path) == [0] and a == 0 and bonus == 1
    ref = O.accept_sample(_tree([9, 3, 2], [-1, 0, 0]), rows, 1.0, u[:, [0, 2, 2, 3]], 3)
    assert ref[1] == 0 and ref[2] == bonus
