"""Pins of the oracle's sampled decoding (speculative sampling, the acceptance
rule of §4.1 at temperature > 0), each against something other than the
oracle itself:

- the inverse-CDF draw equals numpy's searchsorted over the cumulative sum
  (the textbook definition), with its margin, on weights with zeros;
- the tempered distribution equals scipy's softmax of z / T;
- one acceptance test emits tokens distributed exactly as the target p,
  whatever the draft distribution q (the defining property of speculative
  sampling), integrated over fine grids of both uniforms;
- a whole round's first emitted token follows the full model's tempered
  distribution (chi-square over 3000 seeds), while its first draft follows
  the exit distribution; the same statistic rejects the exit distribution
  for the emitted tokens, so the test has power;
- at l* = L the draft and target distributions coincide and every draft is
  kept;
- as the temperature goes to 0 the sampled rounds emit the greedy tokens;
- autoregressive sampling equals numpy's inverse CDF of scipy's softmax at
  the uniforms keyed by position (independent forward passes per token).
"""
import numpy as np
import pytest

import oracle
import synth
from synth.workloads import ModelShape

# Two layers, vocabulary 32, weights large enough that the exit distribution
# at layer 1 is far from the full model's (total variation about 0.5).
MICRO = ModelShape("micro", 2, 64, 2, 2, 32, 128, 32, 1e-5, 10000.0, "f32", sigma=0.1,
                   late_scale=1.0)


@pytest.fixture(scope="module")
def micro():
    om = oracle.Model(MICRO)
    s = om.session(128)
    yield om, s
    s.close()
    om.close()


def test_draw_is_inverse_cdf():
    rng = np.random.default_rng(0)
    for trial in range(50):
        V = int(rng.integers(1, 40))
        w = rng.random(V) * (rng.random(V) < 0.7)
        if w.sum() == 0:
            w[int(rng.integers(V))] = 0.3
        if trial % 2:
            w = w / w.sum()
        W = w.sum()
        C = np.cumsum(w)
        for u in rng.random(20):
            t, mg = oracle.draw(w, u)
            ref = int(np.searchsorted(C, u * W, side="right"))
            assert t == ref, (w, u)
            assert w[t] > 0
            lo = C[t - 1] if t else 0.0
            assert mg == pytest.approx(min(u * W - lo, C[t] - u * W) / W, abs=1e-12)


def test_draw_degenerate_cases():
    assert oracle.draw(np.zeros(5), 0.5)[0] == -1
    one = np.zeros(7)
    one[4] = 2.0
    for u in (1e-7, 0.5, 1 - 2 ** -24):
        assert oracle.draw(one, u)[0] == 4
    # u W at the very top of the mass: the last token of positive weight
    w = np.array([0.0, 0.25, 0.75, 0.0])
    assert oracle.draw(w, 1.0)[0] == 2


def test_tempered_is_softmax():
    from scipy.special import softmax
    rng = np.random.default_rng(1)
    for T in (0.1, 0.6, 1.0, 3.0):
        z = rng.normal(size=300) * 4
        assert np.allclose(oracle.tempered(z, T), softmax(z / T), rtol=1e-12, atol=1e-15)


def _emitted_distribution(p, q, n=2048):
    """P(emitted token) of one acceptance test: the draft d ~ q weighted
    exactly, the two uniforms r and u integrated by the midpoint rule."""
    V = p.size
    grid = (np.arange(n) + 0.5) / n
    out = np.zeros(V)
    kept_frac = np.zeros(V)
    for d in range(V):
        if q[d] == 0:
            continue
        kept = 0
        res = np.zeros(V)
        for r in grid:
            t, ok, am, _ = oracle.spec_step(p, q, d, r, 0.5)
            if ok:
                kept += 1
                assert t == d and am > 0
            else:
                assert am <= 0
        kept_frac[d] = kept / n
        if kept < n:
            for u in grid:
                t, ok, _, _ = oracle.spec_step(p, q, d, 1 - 0.5 / n, u)
                if not ok:
                    res[t] += 1.0 / n
        out[d] += q[d] * kept_frac[d]
        out += q[d] * (1 - kept_frac[d]) * res
    return out, kept_frac


def test_acceptance_rule_keeps_target_distribution():
    rng = np.random.default_rng(2)
    n = 2048
    cases = []
    for _ in range(3):
        p = rng.random(6) ** 3
        q = rng.random(6) ** 3
        cases.append((p / p.sum(), q / q.sum()))
    # q drafts a token p never emits; p has mass where q has none
    cases.append((np.array([0.5, 0.5, 0.0, 0.0]), np.array([0.0, 0.25, 0.25, 0.5])))
    # identical distributions: every draft kept
    cases.append((np.array([0.1, 0.2, 0.7]), np.array([0.1, 0.2, 0.7])))
    for p, q in cases:
        dist, kept = _emitted_distribution(p, q, n)
        # each step function of r or u has at most V jumps: grid error <= V / n
        assert np.abs(dist - p).max() <= p.size / n, (p, q, dist)
        ratio = np.minimum(1.0, np.divide(p, q, out=np.ones_like(p), where=q > 0))
        assert np.abs(kept - ratio)[q > 0].max() <= 1.0 / n


def _chi2(counts, probs, n):
    """Pearson statistic over bins grouped (in order of probability) to an
    expected count of at least 5; returns (statistic, 0.999 quantile)."""
    from scipy import stats
    order = np.argsort(probs)
    E, O = [], []
    ea = oa = 0.0
    for e, c in zip(probs[order] * n, counts[order]):
        ea += e
        oa += c
        if ea >= 5:
            E.append(ea)
            O.append(oa)
            ea = oa = 0.0
    if ea > 0:
        E[-1] += ea
        O[-1] += oa
    E, O = np.array(E), np.array(O)
    return float(((O - E) ** 2 / E).sum()), float(stats.chi2.ppf(0.999, len(E) - 1))


def test_round_emits_target_distribution(micro):
    om, s = micro
    T, N = 0.6, 3000
    ids = synth.prompt_ids(8, MICRO.vocab)
    x = s.prefill(ids)
    seq = list(ids) + [x]
    z, _ = om.exit_head(s.forward(seq, 0, 0, 2)[-1])
    zl, _ = om.exit_head(s.forward(seq, 0, 0, 1)[-1])
    p, q = oracle.tempered(z, T), oracle.tempered(zl, T)
    assert 0.5 * np.abs(p - q).sum() > 0.3  # far apart, so the test has power
    emitted, drafted = np.zeros(MICRO.vocab), np.zeros(MICRO.vocab)
    for seed in range(N):
        s.prefill(ids)
        P = oracle.make_policy(oracle.POLICY_STATIC, kmax=3, static_l=1, static_k=3,
                               temperature=T, sample_seed=seed)
        lg = s.round(P, 8)
        assert lg["sampled"] and lg["pos"] == len(ids)
        emitted[lg["emitted"][0]] += 1
        drafted[lg["drafts"][0]] += 1
    stat, crit = _chi2(emitted, p, N)
    assert stat < crit, (stat, crit)
    stat, crit = _chi2(drafted, q, N)
    assert stat < crit, (stat, crit)
    stat, crit = _chi2(emitted, q, N)
    assert stat > 10 * crit, (stat, crit)


def test_full_depth_exit_keeps_every_sampled_draft(micro):
    om, s = micro
    ids = synth.prompt_ids(8, MICRO.vocab)
    s.prefill(ids)
    P = oracle.make_policy(oracle.POLICY_STATIC, kmax=4, static_l=2, static_k=4, temperature=0.8,
                           sample_seed=3)
    out, logs = s.generate(P, 60)
    assert all(lg["a"] == lg["k"] for lg in logs)
    assert all(m > 0 for lg in logs for m in lg["accept_margin"])


def test_zero_temperature_limit_is_greedy(micro):
    om, s = micro
    ids = synth.prompt_ids(8, MICRO.vocab)
    qp = synth.qnet_hidden_params(3, 16, seed=2)
    mk = lambda T: oracle.make_policy(oracle.POLICY_LEDE, (1, 2), kmax=4, q_params=qp,
                                      q_hidden=16, temperature=T, sample_seed=9)
    s.prefill(ids)
    greedy, glogs = s.generate(mk(0.0), 48)
    # every greedy decision has a top-1/top-2 logit gap of at least 50 T
    # (T = 1e-4), so at T the runner-up weighs below e^-50 of the top token
    gaps = [m for lg in glogs for m in lg["draft_margin"] + lg["verify_margin"]]
    assert min(gaps) > 50e-4
    assert not any(lg["sampled"] for lg in glogs)
    s.prefill(ids)
    sampled, slogs = s.generate(mk(1e-4), 48)
    assert all(lg["sampled"] for lg in slogs)
    assert np.array_equal(greedy, sampled)


def test_sampled_prefill_draws_from_full_model(micro):
    om, s = micro
    T, N = 1.0, 1500
    ids = synth.prompt_ids(8, MICRO.vocab)
    z, _ = om.exit_head(s.forward(ids, 0, 0, 2)[-1])
    p = oracle.tempered(z, T)
    counts = np.zeros(MICRO.vocab)
    for seed in range(N):
        counts[s.prefill(ids, temperature=T, seed=seed)] += 1
    stat, crit = _chi2(counts, p, N)
    assert stat < crit, (stat, crit)
    assert s.prefill(ids) == int(np.argmax(z))


def test_ar_sampling_equals_numpy_restatement(micro):
    """Autoregressive decoding at T = 0.7: every token is numpy's inverse
    CDF (searchsorted over the cumulative sum of scipy's softmax(z / T)) at
    the uniform keyed by (seed, position of the row's input token, purpose
    2, index 0), with z from an independent full-prefix forward pass; the
    token after the prompt uses the key of the last prompt position."""
    from scipy.special import softmax
    om, s = micro
    T, seed, n = 0.7, 21, 24
    ids = list(synth.prompt_ids(8, MICRO.vocab))
    first = s.prefill(ids, temperature=T, seed=seed)
    out, logs = s.generate(oracle.make_policy(oracle.POLICY_AR, temperature=T, sample_seed=seed), n)
    toks = [first] + [int(t) for t in out]
    seq = ids + toks
    checked = 0
    for j, tok in enumerate(toks):
        pre = seq[:len(ids) + j]  # the row that chose tok reads pre[-1]
        z, _ = om.exit_head(s.forward(pre, 0, 0, MICRO.n_layers)[-1])
        C = np.cumsum(softmax(z / T))
        u = float(synth.sample_uniforms(seed, len(pre) - 1, 2, 1)[0])
        ref = int(np.searchsorted(C, u * C[-1], side="right"))
        lo = C[ref - 1] if ref else 0.0
        if min(u * C[-1] - lo, C[ref] - u * C[-1]) > 1e-9:
            assert tok == ref, j
            checked += 1
    assert len(logs) == n and checked >= n - 2
