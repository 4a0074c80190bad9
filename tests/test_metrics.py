"""The acceptance statistics and speedup model of the paper's metrics
(Sec. 5.1): tau, n-alpha of chain drafts, the acceptance rate, omega and
Eq. 9, against closed forms and a simulation of independent acceptances."""
import numpy as np
import pytest

from paper_2505_14260_gb300 import metrics as M


def test_tau_counts_the_added_token():
    assert M.tau([0, 2, 5]) == pytest.approx((1 + 3 + 6) / 3)
    with pytest.raises(ValueError):
        M.tau([])


def test_n_alpha_and_rate_on_hand_counts():
    a = [0, 1, 1, 3, 3, 2]      # chain of depth 3
    # position 1 reached by all 6 and passed by 5; position 2 reached by 5,
    # passed by 3; position 3 reached by 3, passed by 2
    assert M.n_alpha(a, 3) == [5 / 6, 3 / 5, 2 / 3]
    # checked: 0 -> 1, 1 -> 2, 1 -> 2, 3 -> 3, 3 -> 3, 2 -> 3 (14); accepted 10
    assert M.acceptance_rate(a, 3) == pytest.approx(10 / 14)
    assert M.n_alpha([0, 0], 3) == [0.0, None, None]


def test_omega_closed_form():
    for g in range(0, 8):
        for al in (0.0, 0.3, 0.77, 1.0):
            assert M.omega(g, al) == pytest.approx(sum(al ** i for i in range(g + 1)))
    with pytest.raises(ValueError):
        M.omega(3, 1.5)


def test_independent_acceptances_reproduce_omega_and_alpha():
    """Chains whose drafts are accepted independently with probability alpha:
    every n-alpha and the acceptance rate estimate alpha, and tau estimates
    omega(gamma, alpha)."""
    rng = np.random.default_rng(0)
    gamma, alpha, n = 6, 0.6, 200000
    ok = rng.random((n, gamma)) < alpha
    a = np.where(ok.all(1), gamma, np.argmin(ok, axis=1))
    rates = M.n_alpha(a.tolist(), gamma)
    assert all(abs(r - alpha) < 0.01 for r in rates), rates
    assert abs(M.acceptance_rate(a.tolist(), gamma) - alpha) < 0.005
    assert abs(M.tau(a.tolist()) - M.omega(gamma, alpha)) < 0.01


def test_speedup_ratio_limits():
    # no prefill: SR = tokens per cycle x T_p / cycle time
    assert M.speedup_ratio(85, 2.0, 0.0, 2.0, 3.5) == pytest.approx(3.5)
    assert M.speedup_ratio(85, 2.0, 0.0, 4.0, 3.5) == pytest.approx(1.75)
    # prefill dominates: SR -> 1
    assert M.speedup_ratio(1, 2.0, 1e9, 4.0, 3.5) == pytest.approx(1.0, abs=1e-6)
