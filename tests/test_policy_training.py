"""Offline DQN training of the exit policy (§3.2 with the §4.1 schedule) on
walk tables whose optimal policy is known, and the export layout the C ABI
reads.  CPU only: the experience table here is synthetic; collection from
the CUDA path is covered by the GPU tests."""
import numpy as np
import pytest

import oracle
from paper_2606_03113_gb300 import policy as P


def _table(seed=0, n=800):
    """Positions whose exit token becomes correct from candidate j* on; the
    entropy falls through a fixed level exactly there, so 'exit once H <= 5'
    is optimal and learnable from the state."""
    rng = np.random.default_rng(seed)
    cands = (4, 8, 12, 16, 20, 24, 28)
    J = len(cands)
    jstar = rng.integers(0, J + 1, n)  # J: never correct
    j = np.arange(J)[None, :]
    ent = 5.0 + 1.5 * (jstar[:, None] - j) + rng.normal(0, 0.3, (n, J))
    return P.ExitTable(cands, 32, ent + 1.0, ent, rng.uniform(1, 4, n), j >= jstar[:, None])


def test_reward_and_hindsight_bound():
    t = _table()
    # §3.1.3: exit correct 1 + (L - l)/L, wrong -2 + (L - l)/L
    i = int(np.argmax(t.correct[:, 0]))
    assert t.correct[i, 0] and P.walk_reward(t, i, 0) == pytest.approx(1 + 28 / 32)
    i = int(np.argmin(t.correct[:, 6]))
    assert not t.correct[i, 6] and P.walk_reward(t, i, 6) == pytest.approx(-2 + 4 / 32)
    # the hindsight bound dominates every fixed exit index
    ub = P.oracle_walk_return(t)
    for jj in range(7):
        fixed = np.mean([P.walk_reward(t, k, jj) + P.R_CONTINUE * jj for k in range(t.n)])
        assert ub >= fixed


def test_dqn_learns_the_exit_rule():
    t = _table()
    params, st, log = P.train_policy(t, 64, episodes=30000, seeds=(0, 2))
    always_last = np.mean([P.walk_reward(t, k, 6) + 6 * P.R_CONTINUE for k in range(t.n)])
    ub = P.oracle_walk_return(t)
    # far above the forced-exit baseline, most of the way to the hindsight bound
    assert st["mean_return"] > always_last + 0.15, (st, always_last, ub)
    assert st["mean_return"] > 0.75 * ub, (st, ub)
    # exits are correct wherever a correct exit exists (1/8 of positions never have one)
    assert st["correct"] >= np.mean(t.correct.any(axis=1)) - 0.02
    assert len(log.mean_return) >= 2 and log.mean_return[-1] > log.mean_return[0]


def test_export_layout_matches_the_oracle_qnet():
    """The exported parameters, read by the oracle's Q-network in the C ABI
    layout (W1[H][3], b1[H], W2[2][H], b2[2]), give the trained network's
    noise-free values on raw (unstandardised) states."""
    t = _table(1, 200)
    rng = np.random.default_rng(3)
    flat = t.states().reshape(-1, 3)
    net = P.NoisyMLP(16, 0.1, rng, flat.mean(axis=0), flat.std(axis=0))
    params = net.export()
    for s in flat[:20]:
        q_ref = net.q(s[None, :], noisy=False)[0]
        q_orc = oracle.qnet(params, 16, s)
        assert np.allclose(q_orc, q_ref, rtol=1e-4, atol=1e-4)


def test_exit_table_save_and_load_round_trip(tmp_path):
    from paper_2606_03113_gb300.policy import ExitTable
    rng = np.random.default_rng(3)
    t = ExitTable((4, 8, 12), 16, rng.random((50, 3)), rng.random((50, 3)), rng.random(50),
                  rng.random((50, 3)) < 0.4)
    path = str(tmp_path / "table.npz")
    t.save(path)
    u = ExitTable.load(path)
    assert u.cands == t.cands and u.n_layers == t.n_layers
    for name in ("conf", "ent", "trace", "correct"):
        assert np.array_equal(getattr(u, name), getattr(t, name)), name
    assert u.correct.dtype == bool and np.array_equal(u.agreement(), t.agreement())


def test_feature_separation_auc():
    """ExitTable.separation: a feature that orders every correct exit before
    every incorrect one scores 1, its reverse 0, a constant 0.5 (ties count
    one half), and an unrelated feature about 0.5."""
    rng = np.random.default_rng(3)
    n = 400
    correct = rng.random((n, 3)) < 0.5
    conf = np.where(correct, 1.0, 2.0)           # column 0: lower C_5 exactly when correct
    conf[:, 1] = np.where(correct[:, 1], 2.0, 1.0)  # column 1: the reverse
    conf[:, 2] = rng.random(n)                    # column 2: unrelated
    ent = np.full((n, 3), 0.7)                    # constant
    t = P.ExitTable((4, 8, 12), 16, conf, ent, np.zeros(n), correct)
    sep = t.separation()
    assert sep[4]["conf"] == pytest.approx(1.0)
    assert sep[8]["conf"] == pytest.approx(0.0)
    assert abs(sep[12]["conf"] - 0.5) < 0.08
    assert all(v["ent"] == pytest.approx(0.5) for v in sep.values())
