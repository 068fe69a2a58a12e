"""Pins for the CPU oracle: closed forms, hand-built models whose outputs are
known exactly, and the invariants the method fixes (greedy self-speculative
decoding is lossless; exiting at the last layer accepts every draft; the
acceptance count is what independent full-prefix passes give).

Each hand-built case is chosen so that a plausible mistake fails it: the RoPE
pairing and sign, the attention scale, the GQA head mapping, the gate/up
order of SwiGLU, the norm epsilon and weight, the Q-network layout and its tie
rule, the forced exit, and the round's acceptance/rollback bookkeeping.  On
the tiny configuration itself, the oracle's logits at exits 1, 2 and 4 equal a
numpy restatement of the whole decoder within 1e-9 (and on a bf16
grouped-query member of the Llama-3 family).
"""
import math

import numpy as np
import pytest

import oracle
import synth
from synth.workloads import ModelShape, TINY


def hand_shape(L=1, d=4, Hq=1, Hkv=1, hd=4, F=1, V=4, eps=0.0, theta=10000.0):
    return ModelShape("hand", L, d, Hq, Hkv, hd, F, V, eps, theta, "f32", sigma=0.0, late_scale=1.0)


def zeros_model(shape):
    return oracle.Model(shape, synth=False)


# ----------------------------------------------------------------- statistics

def test_stats_uniform_distribution():
    # uniform P over V tokens: H = C_k = ln V, pmax = 1/V, argmax = lowest id
    for V in (5, 1024, 32000):
        st = oracle.stats_from_logits(np.full(V, 0.37), topk=5)
        assert st["entropy"] == pytest.approx(math.log(V), rel=1e-12)
        assert st["conf_k"] == pytest.approx(math.log(V), rel=1e-12)
        assert st["pmax"] == pytest.approx(1.0 / V, rel=1e-12)
        assert st["argmax"] == 0 and st["top_idx"] == [0, 1, 2, 3, 4]
        assert st["margin"] == 0.0


def test_stats_dyadic_distribution():
    # P = (1/2, 1/8, 1/8, 1/8, 1/8): H = 2 ln 2, C_5 = (13/5) ln 2, pmax = 1/2
    p = np.array([0.125, 0.5, 0.125, 0.125, 0.125])
    st = oracle.stats_from_logits(np.log(p) + 3.0, topk=5)
    assert st["entropy"] == pytest.approx(2 * math.log(2), rel=1e-12)
    assert st["conf_k"] == pytest.approx(13 / 5 * math.log(2), rel=1e-12)
    assert st["pmax"] == pytest.approx(0.5, rel=1e-12)
    assert st["argmax"] == 1 and st["top_idx"] == [1, 0, 2, 3, 4]
    assert st["margin"] == pytest.approx(math.log(4), rel=1e-12)
    # C_2 over (1/2, 1/8): (ln 2 + 3 ln 2)/2
    st2 = oracle.stats_from_logits(np.log(p), topk=2)
    assert st2["conf_k"] == pytest.approx(2 * math.log(2), rel=1e-12)


def test_stats_shift_and_permutation_invariance_and_large_logits():
    rng = np.random.default_rng(0)
    z = rng.normal(size=777)
    a = oracle.stats_from_logits(z)
    b = oracle.stats_from_logits(z + 1000.0)  # no overflow, same distribution
    for key in ("entropy", "conf_k", "pmax", "margin"):
        assert a[key] == pytest.approx(b[key], rel=1e-9, abs=1e-12)
    perm = rng.permutation(777)
    c = oracle.stats_from_logits(z[perm])
    assert c["entropy"] == pytest.approx(a["entropy"], rel=1e-12)
    assert perm[c["argmax"]] == a["argmax"]
    # near one-hot: H -> 0, pmax -> 1
    z1 = np.zeros(100)
    z1[7] = 60.0
    d = oracle.stats_from_logits(z1)
    assert d["argmax"] == 7 and d["pmax"] == pytest.approx(1.0, abs=1e-20)
    assert 0.0 <= d["entropy"] < 1e-20


# ---------------------------------------------------------------- trace / Q

def test_trace_confidence_window():
    m = zeros_model(hand_shape())
    s = m.session(8)
    assert s.trace_conf(20) == 0.0
    for _ in range(3):
        s.trace_push(0.25)
    assert s.trace_conf(20) == pytest.approx(math.log(4), rel=1e-12)  # mean over 3 < T
    for _ in range(50):
        s.trace_push(0.5)
    for _ in range(20):
        s.trace_push(0.125)
    assert s.trace_conf(20) == pytest.approx(math.log(8), rel=1e-12)  # only the last T count
    assert s.trace_conf(40) == pytest.approx((math.log(8) * 20 + math.log(2) * 20) / 40, rel=1e-12)


def test_qnet_hand_weights_and_layout():
    # hidden 2: W1 = [[1,0,0],[0,-1,0]], b1 = [0, 0.5], W2 = [[1,1],[2,0]], b2 = [0.1,-0.1]
    P = np.array([1, 0, 0, 0, -1, 0, 0, 0.5, 1, 1, 2, 0, 0.1, -0.1], dtype=np.float32)
    q = oracle.qnet(P, 2, [2.0, 1.0, 7.0])
    # h = relu([2, -0.5]) = [2, 0]; Q = [2 + 0.1, 4 - 0.1]
    assert q[0] == pytest.approx(2.1, abs=1e-6) and q[1] == pytest.approx(3.9, abs=1e-6)
    q2 = oracle.qnet(P, 2, [-1.0, -3.0, 0.0])  # h = relu([-1, 3.5]) = [0, 3.5]
    assert q2[0] == pytest.approx(3.5 + 0.1, abs=1e-6) and q2[1] == pytest.approx(-0.1, abs=1e-6)


# ------------------------------------------------------------ hand-built blocks

def test_rmsnorm_eps_and_weight_through_head():
    sh = hand_shape(eps=0.75)
    m = zeros_model(sh)
    m.set(oracle.T_LMHEAD, 0, np.eye(4))
    m.set(oracle.T_FINAL_NORM, 0, [2.0, 1.0, 1.0, 1.0])
    z = m.logits([3.0, 0.0, 0.0, 0.0])
    # mean(x^2) = 9/4; 3 / sqrt(9/4 + 3/4) * 2 = 2 sqrt(3)
    assert np.allclose(z, [2 * math.sqrt(3), 0, 0, 0], rtol=1e-14, atol=0)


@pytest.mark.parametrize("i,pos", [(0, 1), (0, 5), (1, 2), (1, 700)])
def test_rope_pairing_sign_and_frequency(i, pos):
    sh = hand_shape(theta=10000.0)  # hd = 4: pairs (0,2) and (1,3); inv_freq = 1, 0.01
    m = zeros_model(sh)
    emb = np.zeros((4, 4))
    emb[0, 0] = 3.0  # normalises to 2 e_0 (eps = 0)
    m.set(oracle.T_EMBED, 0, emb)
    w = np.zeros((12, 4))
    w[4 + i, 0] = 0.5  # k = e_i
    m.set(oracle.T_WQKV, 0, w)
    s = m.session(pos + 2)
    s.forward(np.zeros(pos + 1, dtype=np.int32), 0, 0, 1)
    k = [s.kv(0, 0, 0, pos, j) for j in range(4)]
    t = pos * (1.0 if i == 0 else 0.01)
    want = [0.0] * 4
    want[i], want[i + 2] = math.cos(t), math.sin(t)
    assert np.allclose(k, want, rtol=0, atol=1e-12)


def test_attention_softmax_scale_and_causality():
    sh = hand_shape(theta=1e300)  # pair (1,3) effectively unrotated
    m = zeros_model(sh)
    emb = np.zeros((4, 4))
    emb[0, 0] = 3.0  # token 0 -> xhat = 2 e_0
    emb[1, 1] = 3.0  # token 1 -> xhat = 2 e_1
    m.set(oracle.T_EMBED, 0, emb)
    w = np.zeros((12, 4))
    c = 2 * math.log(3)
    w[1, 1] = c / 2       # q(token 1) = c e_1
    w[4 + 1, 0] = 0.5     # k(token 0) = e_1, k(token 1) = 0
    w[8:12, :] = 0.5 * np.eye(4)  # v = xhat / 2 = e_tok
    m.set(oracle.T_WQKV, 0, w)
    m.set(oracle.T_WO, 0, np.eye(4))
    s = m.session(4)
    h = s.forward([0, 1], 0, 0, 1)
    # row 0 sees one key: att = v_0 = e_0; row 1: scores (c*1/sqrt(4), 0) = (ln 3, 0)
    assert np.allclose(h[0], [4, 0, 0, 0], atol=1e-14)
    assert np.allclose(h[1], [0.75, 3.25, 0, 0], atol=1e-12)
    # causality: a different later token leaves row 0 unchanged
    s2 = m.session(4)
    h2 = s2.forward([0, 0], 0, 0, 1)
    assert np.array_equal(h2[0], h[0])


def test_gqa_head_mapping():
    sh = hand_shape(d=8, Hq=4, Hkv=2, hd=2, V=8)
    m = zeros_model(sh)
    m.set(oracle.T_EMBED, 0, np.ones((8, 8)))  # xhat = ones
    w = np.zeros((16, 8))  # q rows 0..7 (zero), k rows 8..11, v rows 12..15
    for j, val in enumerate([1.0, 2.0, 3.0, 4.0]):
        w[12 + j, :] = val / 8.0
    m.set(oracle.T_WQKV, 0, w)
    m.set(oracle.T_WO, 0, np.eye(8))
    s = m.session(2)
    h = s.forward([0], 0, 0, 1)
    # query heads 0,1 read KV head 0 = (1,2); heads 2,3 read KV head 1 = (3,4)
    assert np.allclose(h[0], 1.0 + np.array([1, 2, 1, 2, 3, 4, 3, 4]), atol=1e-13)


def test_swiglu_gate_up_order_and_residual():
    sh = hand_shape(F=2)
    m = zeros_model(sh)
    m.set(oracle.T_EMBED, 0, np.ones((4, 4)))  # xhat = ones
    wgu = np.zeros((4, 4))
    wgu[0, :] = math.log(3) / 4  # gate_0 = ln 3
    wgu[2, :] = 2.0 / 4          # up_0 = 2
    wgu[3, :] = 1.0 / 4          # up_1 = 1, gate_1 = 0 -> silu(0) = 0
    m.set(oracle.T_WGU, 0, wgu)
    wd = np.zeros((4, 2))
    wd[0, 0] = 1.0
    wd[1, 1] = 1.0
    m.set(oracle.T_WDOWN, 0, wd)
    s = m.session(2)
    h = s.forward([0], 0, 0, 1)
    # silu(ln 3) = ln 3 / (1 + 1/3) = 0.75 ln 3; times up = 2
    assert np.allclose(h[0], [1 + 1.5 * math.log(3), 1, 1, 1], atol=1e-14)


def test_identity_layers_accept_everything():
    # zero layer weights: every exit sees the same distribution, so every draft
    # is accepted; identity embedding/head make the greedy token repeat.
    sh = hand_shape(L=4, d=8, Hq=2, Hkv=2, hd=4, F=4, V=8, eps=1e-6)
    m = zeros_model(sh)
    m.set(oracle.T_EMBED, 0, np.eye(8))
    m.set(oracle.T_LMHEAD, 0, np.eye(8))
    s = m.session(64)
    assert s.prefill([1, 2, 3, 5]) == 5
    P = oracle.make_policy(oracle.POLICY_STATIC, kmax=4, static_l=1, static_k=4)
    out, logs = s.generate(P, 12)
    assert list(out) == [5] * 12
    assert all(lg["a"] == lg["k"] for lg in logs)


# ------------------------------------------------------- synthetic weights

def test_late_layer_scaling_statistics():
    w = TINY
    m = oracle.Model(w.shape)
    n = 4096
    for layer, expect in ((1, w.shape.sigma), (2, w.shape.sigma * w.shape.late_scale)):
        vals = np.array([m.get(oracle.T_WO, layer, i) for i in range(n)])
        assert abs(vals.std() / expect - 1) < 0.05
    # first element of layer-0 wqkv equals the generator's value (same stream)
    g = synth.weights_f32(0, 16 + 0, 0, 4, w.shape.sigma)
    assert [m.get(oracle.T_WQKV, 0, i) for i in range(4)] == [float(x) for x in g]


# --------------------------------------------------------- generation pins

def lede_policy(w, qp, kmax=None):
    return oracle.make_policy(oracle.POLICY_LEDE, w.candidates, kmax=kmax or w.kmax,
                              q_params=qp, q_hidden=w.qnet_hidden)


def fixed_q(hidden, q_cont, q_exit):
    p = np.zeros(hidden * 3 + hidden + 2 * hidden + 2, dtype=np.float32)
    p[-2], p[-1] = q_cont, q_exit
    return p


@pytest.fixture(scope="module")
def tiny_setup():
    w = TINY
    m = oracle.Model(w.shape)
    ids = synth.prompt_ids(w.prompt_len, w.shape.vocab)
    return w, m, ids


def generate(w, m, ids, policy, n):
    s = m.session(w.max_seq)
    first = s.prefill(ids)
    out, logs = s.generate(policy, n)
    return first, out, logs


@pytest.mark.parametrize("seed", [2, 7, 11])
def test_ssd_equals_ar_any_policy(tiny_setup, seed):
    w, m, ids = tiny_setup
    _, ar, _ = generate(w, m, ids, oracle.make_policy(oracle.POLICY_AR), 40)
    qp = synth.qnet_hidden_params(3, w.qnet_hidden, seed=seed)
    _, le, logs = generate(w, m, ids, lede_policy(w, qp), 40)
    assert np.array_equal(ar, le)
    assert sum(lg["n_emit"] for lg in logs) == 40
    for l, k in ((1, 1), (2, 3), (3, 4)):
        _, st, _ = generate(w, m, ids, oracle.make_policy(oracle.POLICY_STATIC, kmax=w.kmax,
                                                          static_l=l, static_k=k), 40)
        assert np.array_equal(ar, st)


def test_exit_at_last_layer_accepts_every_draft(tiny_setup):
    w, m, ids = tiny_setup
    L = w.shape.n_layers
    _, _, logs = generate(w, m, ids, oracle.make_policy(oracle.POLICY_STATIC, kmax=4, static_l=L,
                                                        static_k=4), 30)
    assert all(lg["a"] == lg["k"] for lg in logs)
    assert all(lg["lstar"] == L for lg in logs if lg["k"] > 0)
    # same through the learned-policy path with a single candidate {L}
    P = oracle.make_policy(oracle.POLICY_LEDE, (L,), kmax=4, q_params=fixed_q(8, 0.0, 1.0),
                           q_hidden=8)
    _, _, logs = generate(w, m, ids, P, 30)
    assert all(lg["a"] == lg["k"] and lg["k"] == lg["kcap"] for lg in logs)


def test_walk_semantics_fixed_q(tiny_setup):
    w, m, ids = tiny_setup
    c = list(w.candidates)
    # always continue: walk to the last candidate (forced exit), stop after d_1
    for qc, qe in ((1.0, 0.0), (0.5, 0.5)):  # a tie counts as continue
        P = oracle.make_policy(oracle.POLICY_LEDE, c, kmax=4, q_params=fixed_q(4, qc, qe), q_hidden=4)
        _, _, logs = generate(w, m, ids, P, 20)
        for lg in logs[:-1]:
            assert lg["visited"] == c and lg["lstar"] == c[-1] and lg["k"] == 1
            assert lg["q_action"] == [0] * len(c)
    # always exit: exit at the first candidate and draft up to kcap
    P = oracle.make_policy(oracle.POLICY_LEDE, c, kmax=4, q_params=fixed_q(4, 0.0, 1.0), q_hidden=4)
    _, _, logs = generate(w, m, ids, P, 20)
    for lg in logs:
        if lg["kcap"] > 0:
            assert lg["visited"] == [c[0]] and lg["lstar"] == c[0] and lg["k"] == lg["kcap"]
    assert logs[-1]["kcap"] == 0 or sum(l["n_emit"] for l in logs) == 20


def test_acceptance_matches_brute_force(tiny_setup):
    """Every draft and every verification token is recomputed by an
    independent pass over the whole prefix on a fresh session."""
    w, m, ids = tiny_setup
    qp = synth.qnet_hidden_params(3, w.qnet_hidden, seed=5)
    P = oracle.make_policy(oracle.POLICY_LEDE, w.candidates, kmax=4, q_params=qp,
                           q_hidden=w.qnet_hidden)
    first, out, logs = generate(w, m, ids, P, 24)
    L = w.shape.n_layers
    seq = list(ids) + [first]
    for lg in logs[:8]:
        prefix = list(seq)  # ends with the pending token x
        assert prefix[-1] == lg["x"] and len(prefix) - 1 == lg["pos"]
        toks = prefix + lg["drafts"]
        for i in range(lg["k"] + 1):
            s = m.session(w.max_seq)
            h = s.forward(toks[:len(prefix) + i], 0, 0, L)
            _, st = m.exit_head(h[-1])
            assert st["argmax"] == lg["verify_tok"][i]
        for i in range(lg["k"]):
            s = m.session(w.max_seq)
            h = s.forward(toks[:len(prefix) + i], 0, 0, lg["lstar"])
            _, st = m.exit_head(h[-1])
            assert st["argmax"] == lg["drafts"][i]
        a = 0
        while a < lg["k"] and lg["drafts"][a] == lg["verify_tok"][a]:
            a += 1
        assert a == lg["a"] and lg["emitted"] == lg["drafts"][:a] + [lg["verify_tok"][a]]
        seq += lg["emitted"]


def test_round_bookkeeping_and_resume(tiny_setup):
    w, m, ids = tiny_setup
    qp = synth.qnet_hidden_params(3, w.qnet_hidden, seed=3)
    P = lede_policy(w, qp)
    s = m.session(w.max_seq)
    first = s.prefill(ids)
    seq = list(ids) + [first]
    logs = []
    for _ in range(6):
        lg = s.round(P, 64)
        assert s.kv_len == lg["pos"] + lg["a"] + 1 and s.x == lg["emitted"][-1]
        seq += lg["emitted"]
        logs.append(lg)
    # resume from the emitted sequence: the next round is identical bit for bit
    nxt = s.round(P, 64)
    s2 = m.session(w.max_seq)
    s2.resume(seq)
    assert s2.kv_len == s.kv_len - nxt["a"] - 1 and s2.x == nxt["x"]
    again = s2.round(P, 64)
    assert again == nxt
    # Q decisions: each recorded state reproduces its action and values
    for lg in logs:
        for st, qv, act in zip(lg["q_state"], lg["q_val"], lg["q_action"]):
            q = oracle.qnet(qp, w.qnet_hidden, st)
            assert tuple(q) == qv and act == int(q[1] > q[0])


def test_error_paths():
    m = zeros_model(hand_shape())
    s = m.session(4)
    P = oracle.make_policy(oracle.POLICY_AR)
    with pytest.raises(oracle.OracleError):
        s.round(P, 4)  # before prefill
    with pytest.raises(oracle.OracleError):
        s.prefill([0, 1, 2, 3])  # no room for the pending token
    s.prefill([0, 1])
    bad = oracle.make_policy(oracle.POLICY_LEDE, (2, 1), kmax=2, q_params=fixed_q(2, 0, 1), q_hidden=2)
    with pytest.raises(oracle.OracleError):
        s.round(bad, 4)  # candidates must ascend
    with pytest.raises(oracle.OracleError):
        s.forward([9], 0, 0, 1)  # token out of vocabulary


# ------------------------------------------------ policy variants (Table 3, §4.1)

def _rounds(logs):
    return [(lg["lstar"], lg["k"], lg["drafts"], lg["a"], lg["emitted"]) for lg in logs]


@pytest.mark.parametrize("l,f", [(1, 2), (2, 3), (3, 4)])
def test_fixed_length_single_candidate_is_static(tiny_setup, l, f):
    """LEDE without dynamic exit and without adaptive drafting (one candidate,
    fixed length) is exactly the static (l, f) policy, round for round, for
    any Q-network: the only walk decision is a forced exit and the length is
    not asked of the network."""
    w, m, ids = tiny_setup
    qp = synth.qnet_hidden_params(3, w.qnet_hidden, seed=3)
    P = oracle.make_policy(oracle.POLICY_LEDE, (l,), kmax=w.kmax, q_params=qp,
                           q_hidden=w.qnet_hidden, fixed_k=f)
    S = oracle.make_policy(oracle.POLICY_STATIC, kmax=w.kmax, static_l=l, static_k=f)
    _, a, la = generate(w, m, ids, P, 30)
    _, b, lb = generate(w, m, ids, S, 30)
    assert np.array_equal(a, b) and _rounds(la) == _rounds(lb)
    # one Q decision per round (the walk), none after drafts
    assert all(len(lg["q_action"]) == (1 if lg["kcap"] > 0 else 0) for lg in la)


def test_fixed_length_keeps_the_walk(tiny_setup):
    """Without adaptive drafting the walk still chooses l* by the Q-network
    (always exit: the first candidate), and every speculative round drafts
    min(fixed_k, cap) tokens."""
    w, m, ids = tiny_setup
    c = list(w.candidates)
    for qc, qe, lstar in ((0.0, 1.0, c[0]), (1.0, 0.0, c[-1])):
        P = oracle.make_policy(oracle.POLICY_LEDE, c, kmax=4, q_params=fixed_q(4, qc, qe),
                               q_hidden=4, fixed_k=3)
        out, logs = generate(w, m, ids, P, 25)[1:]
        _, ar, _ = generate(w, m, ids, oracle.make_policy(oracle.POLICY_AR), 25)
        assert np.array_equal(out, ar)
        for lg in logs:
            if lg["kcap"] > 0:
                assert lg["lstar"] == lstar and lg["k"] == min(3, lg["kcap"]) == lg["kcap"]


def test_single_candidate_adaptive_drafting(tiny_setup):
    """Without dynamic exit (one candidate), an always-exit Q-network drafts
    to the cap and a never-exit one drafts d_1 only: static (l, kmax) and
    static (l, 1) round for round."""
    w, m, ids = tiny_setup
    for qc, qe, k in ((0.0, 1.0, w.kmax), (1.0, 0.0, 1)):
        P = oracle.make_policy(oracle.POLICY_LEDE, (2,), kmax=w.kmax, q_params=fixed_q(4, qc, qe),
                               q_hidden=4)
        S = oracle.make_policy(oracle.POLICY_STATIC, kmax=w.kmax, static_l=2, static_k=k)
        _, a, la = generate(w, m, ids, P, 30)
        _, b, lb = generate(w, m, ids, S, 30)
        assert np.array_equal(a, b) and _rounds(la) == _rounds(lb)


def test_threshold_limits_and_rule(tiny_setup):
    """Confidence-threshold drafting: a threshold no probability can miss
    drafts to the cap (static (l, kmax)), one none can reach drafts d_1 only
    (static (l, 1)); in between, each logged decision is pmax >= tau and
    drafting stopped exactly at the first failed one or at the cap."""
    w, m, ids = tiny_setup
    pmax_seen = []
    for tau, k in ((1e-12, w.kmax), (1.0, 1)):  # pmax < 1 for any spread distribution
        P = oracle.make_policy(oracle.POLICY_THRESHOLD, kmax=w.kmax, static_l=2, conf_threshold=tau)
        S = oracle.make_policy(oracle.POLICY_STATIC, kmax=w.kmax, static_l=2, static_k=k)
        _, a, la = generate(w, m, ids, P, 30)
        _, b, lb = generate(w, m, ids, S, 30)
        assert np.array_equal(a, b) and _rounds(la) == _rounds(lb)
        if tau < 1.0:
            pmax_seen += [p for lg in la for _, p in lg["q_val"]]
    # a threshold at the median observed draft confidence splits the decisions
    tau = float(np.median(pmax_seen))
    P = oracle.make_policy(oracle.POLICY_THRESHOLD, kmax=w.kmax, static_l=2, conf_threshold=tau)
    out, logs = generate(w, m, ids, P, 40)[1:]
    _, ar, _ = generate(w, m, ids, oracle.make_policy(oracle.POLICY_AR), 40)
    assert np.array_equal(out, ar)
    seen_both = set()
    for lg in logs:
        if lg["kcap"] == 0:
            continue
        acts = lg["q_action"]
        assert len(acts) == lg["k"]  # one decision after each draft
        for a, (t, p) in zip(acts, lg["q_val"]):
            assert t == tau and a == (1 if p >= tau else 0)
            seen_both.add(a)
        stopped = [i for i, a in enumerate(acts) if a == 0]
        assert lg["k"] == (stopped[0] + 1 if stopped else lg["kcap"])
    assert seen_both == {0, 1}  # the threshold actually splits this run's decisions


def test_variant_policies_rejected_when_malformed(tiny_setup):
    w, m, ids = tiny_setup
    s = m.session(w.max_seq)
    s.prefill(ids)
    bad = [oracle.make_policy(oracle.POLICY_THRESHOLD, kmax=4, static_l=2, conf_threshold=0.0),
           oracle.make_policy(oracle.POLICY_THRESHOLD, kmax=4, static_l=2, conf_threshold=1.5),
           oracle.make_policy(oracle.POLICY_THRESHOLD, kmax=4, static_l=0, conf_threshold=0.5),
           oracle.make_policy(oracle.POLICY_LEDE, (1, 2), kmax=4, q_params=fixed_q(4, 0, 1),
                              q_hidden=4, fixed_k=-1)]
    for P in bad:
        with pytest.raises(oracle.OracleError):
            s.round(P, 10)


# ------------------------------------------------ composition on a real shape


def _numpy_forward(shape, ids, l_exit):
    """The Llama decoder of the tiny configuration written out in numpy
    (weights from the seeded generator): pre-RMSNorm blocks with RoPE
    ("rotate half", angle pos * theta^(-2i/hd)), causal GQA attention scaled
    by 1/sqrt(hd), SwiGLU down(silu(gate) * up), the second half's out/down
    projections scaled; then the shared final RMSNorm and LM head on the
    hidden states after l_exit blocks.  Returns logits [n][vocab]."""
    s = shape
    d, hd, Hq, Hkv, F, V = s.d_model, s.head_dim, s.n_heads, s.n_kv_heads, s.ffn_dim, s.vocab

    def mat(tid, rows, cols, sig):
        if s.dtype == "bf16":  # bf16 storage: the generator's values rounded to bf16
            w = synth.bf16_bits_to_f32(
                synth.weights_bf16_bits(synth.SEED_WEIGHTS, tid, 0, rows * cols, sig))
        else:
            w = synth.weights_f32(synth.SEED_WEIGHTS, tid, 0, rows * cols, sig)
        return w.astype(np.float64).reshape(rows, cols)

    def rms(x):
        return x / np.sqrt((x * x).mean(axis=-1, keepdims=True) + s.rms_eps)

    n = len(ids)
    pos = np.arange(n)[:, None]
    ang = pos * s.rope_theta ** (-2.0 * np.arange(hd // 2) / hd)[None, :]
    cos, sin = np.cos(ang), np.sin(ang)

    def rope(v):  # v [n][heads][hd]
        a, b = v[..., :hd // 2], v[..., hd // 2:]
        c, si = cos[:, None, :], sin[:, None, :]
        return np.concatenate([a * c - b * si, a * si + b * c], axis=-1)

    h = mat(synth.TID_EMBED, V, d, s.sigma)[ids]
    for l in range(l_exit):
        late = s.late_scale if l >= s.n_layers // 2 else 1.0
        wqkv = mat(synth.layer_tid(l, 0), (Hq + 2 * Hkv) * hd, d, s.sigma)
        wo = mat(synth.layer_tid(l, 1), d, Hq * hd, s.sigma * late)
        wgu = mat(synth.layer_tid(l, 2), 2 * F, d, s.sigma)
        wdown = mat(synth.layer_tid(l, 3), d, F, s.sigma * late)
        qkv = rms(h) @ wqkv.T
        q = rope(qkv[:, :Hq * hd].reshape(n, Hq, hd))
        k = rope(qkv[:, Hq * hd:(Hq + Hkv) * hd].reshape(n, Hkv, hd))
        v = qkv[:, (Hq + Hkv) * hd:].reshape(n, Hkv, hd)
        out = np.zeros((n, Hq, hd))
        for hq in range(Hq):
            kv = hq // (Hq // Hkv)
            sc = q[:, hq, :] @ k[:, kv, :].T / math.sqrt(hd)
            sc = np.where(np.tril(np.ones((n, n))) > 0, sc, -np.inf)
            p = np.exp(sc - sc.max(axis=1, keepdims=True))
            out[:, hq, :] = (p / p.sum(axis=1, keepdims=True)) @ v[:, kv, :]
        h = h + out.reshape(n, Hq * hd) @ wo.T
        gu = rms(h) @ wgu.T
        g, u = gu[:, :F], gu[:, F:]
        h = h + (g / (1.0 + np.exp(-g)) * u) @ wdown.T
    return rms(h) @ mat(synth.TID_LMHEAD, V, d, s.sigma).T


# a bf16 member of the Llama-3 family: grouped-query attention (4 query heads
# per KV head), theta 500000, bf16 weights and embeddings
SMALL_GQA_BF16 = ModelShape("gqa-bf16", 4, 256, 8, 2, 32, 512, 1024, 1e-5, 500000.0, "bf16",
                            sigma=0.05, late_scale=0.2)


# query width Hq * hd (4 x 24 = 96) unlike d (80), every dimension distinct:
# a transposed projection or a rows/cols mix-up changes every output
ODD_F32 = ModelShape("odd-f32", 4, 80, 4, 2, 24, 56, 72, 1e-5, 10000.0, "f32", sigma=0.05,
                     late_scale=0.3)
ODD_BF16 = ModelShape("odd-bf16", 4, 80, 4, 2, 24, 56, 72, 1e-5, 500000.0, "bf16", sigma=0.05,
                      late_scale=0.3)


@pytest.mark.parametrize("shape,l_exit", [(TINY.shape, 1), (TINY.shape, 2), (TINY.shape, 4),
                                          (SMALL_GQA_BF16, 3), (SMALL_GQA_BF16, 4),
                                          (ODD_BF16, 4)])
def test_numpy_restatement_of_the_tiny_forward(shape, l_exit):
    s = shape
    ids = list(synth.prompt_ids(12, s.vocab))
    ref = _numpy_forward(s, ids, l_exit)
    om = oracle.Model(s)
    try:
        h = om.session(32).forward(ids, 0, 0, l_exit)
        for i in range(len(ids)):
            z = om.logits(h[i])
            assert np.abs(z - ref[i]).max() <= 1e-9 * np.abs(ref[i]).max(), (l_exit, i)
    finally:
        om.close()


# -------------------------------------- matrix products the GPU tests check with


def _generated(s, tid, rows, cols, sig, seed=synth.SEED_WEIGHTS, start=0):
    """Rows of a generated matrix from the seeded generator alone (synth.h),
    in the model's storage precision, as a float64 numpy array."""
    if s.dtype == "bf16":
        w = synth.bf16_bits_to_f32(synth.weights_bf16_bits(seed, tid, start, rows * cols, sig))
    else:
        w = synth.weights_f32(seed, tid, start, rows * cols, sig)
    return w.astype(np.float64).reshape(rows, cols)


def _matrices(s):
    """(selector, tensor id of layer l, rows, cols, late-scaled) of every matrix."""
    d, qd = s.d_model, s.n_heads * s.head_dim
    return [(oracle.T_WQKV, lambda l: synth.layer_tid(l, synth.LT_WQKV), s.qkv_rows, d, False),
            (oracle.T_WO, lambda l: synth.layer_tid(l, synth.LT_WO), d, qd, True),
            (oracle.T_WGU, lambda l: synth.layer_tid(l, synth.LT_WGU), 2 * s.ffn_dim, d, False),
            (oracle.T_WDOWN, lambda l: synth.layer_tid(l, synth.LT_WDOWN), d, s.ffn_dim, True),
            (oracle.T_LMHEAD, lambda l: synth.TID_LMHEAD, s.vocab, d, False),
            (oracle.T_EMBED, lambda l: synth.TID_EMBED, s.vocab, d, False)]


@pytest.mark.parametrize("shape", [ODD_F32, ODD_BF16])
def test_orc_matvec_every_matrix_against_numpy(shape):
    """orc_matvec picks each matrix's own row and column counts: the product
    equals numpy's W @ x with W taken from the generator, for every matrix
    kind, early and late (scaled) layers, on a shape whose query width
    differs from d."""
    s = shape
    om = oracle.Model(s)
    rng = np.random.default_rng(11)
    try:
        for which, tid, rows, cols, late in _matrices(s):
            for l in (0, s.n_layers - 1):
                sig = s.sigma * (s.late_scale if late and l >= s.n_layers // 2 else 1.0)
                W = _generated(s, tid(l), rows, cols, sig)
                x = rng.normal(size=cols)
                y = om.matvec(which, l, x)
                ref = W @ x
                assert y.shape == (rows,)
                assert np.abs(y - ref).max() <= 1e-12 * np.abs(ref).max(), (which, l)
    finally:
        om.close()


@pytest.mark.parametrize("bf16", [False, True])
def test_orc_matvec_synth_against_numpy_and_the_model(bf16):
    """orc_matvec_synth (the checker of the full-size products) takes row
    row0 + r of a K-column generated matrix from flat index (row0 + r) K + k:
    a block of rows away from the start, with K odd, equals numpy's product of
    the generator's rows; and on every matrix of a model it equals the
    model's own product bit for bit (same values, same order)."""
    s = ODD_BF16 if bf16 else ODD_F32
    rng = np.random.default_rng(5)
    seed, tid, sig, K, row0, n = 3, 77, 0.03, 203, 37, 11
    W = _generated(s, tid, n, K, sig, seed=seed, start=row0 * K)
    x = rng.normal(size=K)
    y = oracle.matvec_synth(seed, tid, sig, bf16, row0, n, x)
    assert np.abs(y - W @ x).max() <= 1e-12 * np.abs(W @ x).max()
    # the first row alone, and a different row0, select different rows
    y1 = oracle.matvec_synth(seed, tid, sig, bf16, row0 + 3, 1, x)
    assert y1[0] == y[3]
    om = oracle.Model(s)
    try:
        for which, tid_l, rows, cols, late in _matrices(s):
            for l in (0, s.n_layers - 1):
                sc = s.sigma * (s.late_scale if late and l >= s.n_layers // 2 else 1.0)
                x = rng.normal(size=cols)
                ym = om.matvec(which, l, x)
                ys = oracle.matvec_synth(synth.SEED_WEIGHTS, tid_l(l), sc, bf16, 0, rows, x)
                assert np.array_equal(ym, ys), (which, l)
    finally:
        om.close()


def test_oracle_struct_layouts_match_the_c_compiler(tmp_path):
    """The ctypes mirrors of the oracle's structs match lede_oracle.h field
    by field (a mismatch would silently corrupt every oracle result)."""
    import ctypes
    import os
    import subprocess
    structs = {"orc_cfg": oracle.Cfg, "orc_stats": oracle.Stats, "orc_policy": oracle.Policy,
               "orc_round_log": oracle.RoundLog}
    lines = ['#include <stddef.h>', '#include <stdio.h>', '#include "lede_oracle.h"',
             "int main(void) {"]
    for cname, st in structs.items():
        lines.append(f'  printf("{cname} sizeof %zu\\n", sizeof({cname}));')
        for field, _ in st._fields_:
            lines.append(f'  printf("{cname} {field} %zu\\n", offsetof({cname}, {field}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.check_call(["gcc", "-std=c11", "-I", os.path.dirname(oracle.__file__), str(src),
                           "-o", str(exe)])
    out = subprocess.check_output([str(exe)], text=True).split("\n")
    got = {tuple(l.split()[:2]): int(l.split()[2]) for l in out if l.strip()}
    for cname, st in structs.items():
        assert got[(cname, "sizeof")] == ctypes.sizeof(st), cname
        for field, _ in st._fields_:
            assert got[(cname, field)] == getattr(st, field).offset, (cname, field)
