"""Pins of the oracle's pooled Q-network state (the tiny configuration's
state: the mean over the round's rows so far of the exit hidden state after
the final RMSNorm, then the exit distribution's max-probability; d_model + 1
inputs), against a numpy restatement and hand-set networks:

- a network that reads only the last input decides exit iff pmax > tau and
  logs Q = (tau, pmax) exactly;
- a network that reads one pooled coordinate logs that coordinate, which
  equals numpy's RMSNorm of the full-prefix hidden states (independent
  forward passes), averaged over exactly the rows the reading names: the
  pending token at each walk candidate, the pending token and the drafts so
  far at l* while drafting;
- greedy self-speculative decoding with the pooled state still emits the
  autoregressive tokens;
- the "discard" reading of adaptive drafting (a continue action drops the
  draft it was taken on), against the default "keep" reading, on a network
  whose decisions are known from the logged max-probabilities.
"""
import numpy as np
import pytest

import oracle
import synth
from synth.workloads import TINY

W = TINY
S = W.shape
D = S.d_model


@pytest.fixture(scope="module")
def om():
    m = oracle.Model(S)
    yield m
    m.close()


def _pack(W1, b1, W2, b2):
    return np.concatenate([W1.ravel(), b1, W2.ravel(), b2]).astype(np.float32)


def _policy(qp, H, kmax=4, fixed_k=0):
    return oracle.make_policy(oracle.POLICY_LEDE, W.candidates, kmax=kmax, q_params=qp,
                              q_hidden=H, q_in=D + 1, fixed_k=fixed_k)


def test_pmax_only_network(om):
    tau = 0.004
    W1 = np.zeros((2, D + 1))
    W1[0, D] = 1.0
    b1 = np.array([0.0, 1.0])
    W2 = np.array([[0.0, tau], [1.0, 0.0]])  # rows: Q(continue), Q(exit)
    qp = _pack(W1, b1, W2, np.zeros(2))
    s = om.session(W.max_seq)
    s.prefill(synth.prompt_ids(W.prompt_len, S.vocab))
    _, logs = s.generate(_policy(qp, 2), 40)
    n = 0
    for lg in logs:
        for a, (qc, qe), st in zip(lg["q_action"], lg["q_val"], lg["q_state"]):
            pmax = st[0]
            assert qc == pytest.approx(np.float32(tau), abs=1e-12)
            assert qe == pytest.approx(pmax, abs=1e-12)
            assert a == int(pmax > np.float32(tau))
            n += 1
    assert n >= 40


def _normed_rows(om, tokens, layer, rows):
    """numpy: final RMSNorm of the hidden states at `layer` of the given
    positions, from one full-prefix forward pass of a fresh session."""
    s = om.session(len(tokens) + 1)
    h = s.forward(tokens, 0, 0, layer)
    s.close()
    g = np.array([om.get(oracle.T_FINAL_NORM, 0, i) for i in range(D)])
    x = h[rows]
    return x / np.sqrt((x * x).mean(axis=1, keepdims=True) + S.rms_eps) * g


@pytest.mark.parametrize("coord", [0, 137])
def test_pooled_coordinate_equals_numpy_restatement(om, coord):
    big = 50.0
    W1 = np.zeros((1, D + 1))
    W1[0, coord] = 1.0
    b1 = np.array([big])
    W2 = np.array([[0.0], [1.0]])
    b2 = np.array([0.0, -big])  # Q(exit) = pooled mean[coord], Q(continue) = 0
    qp = _pack(W1, b1, W2, b2)
    ids = list(synth.prompt_ids(W.prompt_len, S.vocab))
    s = om.session(W.max_seq)
    first = s.prefill(ids)
    _, logs = s.generate(_policy(qp, 1), 24)
    seq = ids + [first]
    checked = 0
    for lg in logs[:8]:
        p, x = lg["pos"], lg["x"]
        assert len(seq) == p + 1 and seq[-1] == x
        nv = len(lg["visited"])
        for j, layer in enumerate(lg["visited"]):  # walk: the pending token only
            ref = _normed_rows(om, seq, layer, [p]).mean(axis=0)[coord]
            assert lg["q_val"][j][1] == pytest.approx(ref, rel=1e-9, abs=1e-12)
            assert lg["q_state"][j][1] == 1
            checked += 1
        for i in range(1, lg["k"]):  # after draft i + 1: x, d_1..d_i at l*
            toks = seq + lg["drafts"][:i]
            ref = _normed_rows(om, toks, lg["lstar"], list(range(p, p + i + 1))).mean(axis=0)
            assert lg["q_val"][nv + i - 1][1] == pytest.approx(ref[coord], rel=1e-9, abs=1e-12)
            assert lg["q_state"][nv + i - 1][1] == i + 1
            assert lg["q_state"][nv + i - 1][2] == pytest.approx(np.linalg.norm(ref), rel=1e-9)
            checked += 1
        seq += lg["emitted"]
    assert checked >= 10


@pytest.mark.parametrize("fixed_k", [0, 3])
def test_pooled_state_ssd_equals_ar(om, fixed_k):
    ids = synth.prompt_ids(W.prompt_len, S.vocab)
    s = om.session(W.max_seq)
    s.prefill(ids)
    ar, _ = s.generate(oracle.make_policy(oracle.POLICY_AR), W.gen_len)
    qp = synth.qnet_hidden_params(D + 1, W.qnet_hidden)
    s.prefill(ids)
    out, logs = s.generate(_policy(qp, W.qnet_hidden, fixed_k=fixed_k), W.gen_len)
    assert np.array_equal(ar, out)
    assert sum(lg["k"] for lg in logs) > 0


def test_pooled_state_rejects_other_widths(om):
    qp = synth.qnet_hidden_params(D, 8)
    s = om.session(W.max_seq)
    s.prefill(synth.prompt_ids(8, S.vocab))
    P = oracle.make_policy(oracle.POLICY_LEDE, W.candidates, kmax=4, q_params=qp, q_hidden=8,
                           q_in=D)
    with pytest.raises(oracle.OracleError):
        s.round(P, 8)


# ------------------------------------------------- the "discard" reading


@pytest.mark.parametrize("discard", [False, True])
def test_discard_reading_of_adaptive_drafting(om, discard):
    """With a network that exits iff pmax > tau, the keep reading (default)
    keeps every draft and stops after the first continue; the discard
    reading drops the draft whose decision was continue.  Either way the
    output is the autoregressive one."""
    tau = 0.003
    W1 = np.zeros((2, D + 1))
    W1[0, D] = 1.0
    b1 = np.array([0.0, 1.0])
    W2 = np.array([[0.0, tau], [1.0, 0.0]])
    qp = _pack(W1, b1, W2, np.zeros(2))
    ids = synth.prompt_ids(W.prompt_len, S.vocab)
    s = om.session(W.max_seq)
    s.prefill(ids)
    ar, _ = s.generate(oracle.make_policy(oracle.POLICY_AR), W.gen_len)
    s.prefill(ids)
    P = oracle.make_policy(oracle.POLICY_LEDE, W.candidates, kmax=4, q_params=qp, q_hidden=2,
                           q_in=D + 1, discard_on_continue=discard)
    out, logs = s.generate(P, W.gen_len)
    assert np.array_equal(ar, out)
    dropped = 0
    for lg in logs:
        if lg["kcap"] == 0:
            continue
        nv = len(lg["visited"])
        after = lg["q_action"][nv:]  # decisions taken on drafts 2, 3, ...
        assert all(after[:-1])  # drafting goes on while the action is exit
        stop = len(after) > 0 and after[-1] == 0
        if discard and stop:
            assert lg["k"] == len(after)  # d_1 and the drafts whose action was exit
            dropped += 1
        else:
            assert lg["k"] == 1 + len(after)
    if discard:
        assert dropped >= 3
