"""Host logic of bench.py on the CPU: the algorithmic bytes of a round, the
kernel-launch count of a round graph, the ncu traffic lookup and the clock
record parser."""
import os
import re
import sys

import pytest

REPO = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, REPO)

import bench  # noqa: E402
from paper_2606_03113_gb300.runtime import kernels_per_round, pass_launches  # noqa: E402
from synth.workloads import LLAMA2_7B, TINY  # noqa: E402


def test_round_bytes_worked_example():
    """Llama-2-7B shape, two candidates visited, exit at layer 8, six drafts,
    context about 640: 2 LM heads + 6 partial passes of 8 layers (5 with a
    head) + one full pass with a head, plus the KV of each pass, about
    35.3 GB per round."""
    s = LLAMA2_7B.shape
    tr = dict(pos=637, kcap=12, visited=[4, 8], lstar=8, k=6)
    b = bench.round_bytes(LLAMA2_7B, tr)
    Wl, head = s.layer_weight_bytes(), s.lm_head_bytes()
    assert Wl == 404750336 and head == 262144000
    weights = 2 * head + 6 * 8 * Wl + 5 * head + 32 * Wl + head
    assert weights < b < weights + 1.0e9  # KV: 16 KB per position and layer
    assert b == pytest.approx(35.3e9, rel=0.01)


def test_round_bytes_autoregressive():
    s = LLAMA2_7B.shape
    pos = 700
    tr = dict(pos=pos, kcap=0, visited=[], lstar=0, k=0)
    kv = 2 * s.n_kv_heads * s.head_dim * 2 * (pos + 1)  # K and V rows read per layer
    assert bench.round_bytes(LLAMA2_7B, tr) == s.n_layers * (s.layer_weight_bytes() + kv) \
        + s.lm_head_bytes()


def test_kernel_launches_of_a_round():
    L = LLAMA2_7B.shape.n_layers
    # bf16 pass over n layers: first QKV, then attention + chained launch per layer
    assert [pass_launches(n) for n in (0, 1, 4)] == [0, 3, 9]
    assert pass_launches(4, bf16=False) == 20
    # autoregressive round: round_begin, embed, pass, head, accept
    ar = dict(kcap=0, visited=[], lstar=0, k=0)
    assert kernels_per_round(ar, L, 0) == 1 + 1 + (2 * L + 1) + 1 + 1
    # LEDE round: walk over candidates 4 and 8 (segment pass, head, decide),
    # draft_begin, two further drafts (embed, 8 layers, head, decide), verify
    tr = dict(kcap=12, visited=[4, 8], lstar=8, k=3)
    walk = 1 + (9 + 2) + (9 + 2)
    drafts = 1 + 2 * (1 + 17 + 2)
    verify = 1 + (2 * L + 1) + 1 + 1
    assert kernels_per_round(tr, L, 0) == 1 + walk + drafts + verify
    assert bench.kernels_in_round(LLAMA2_7B, tr) == 1 + walk + drafts + verify
    assert bench.kernels_in_round(TINY, ar) == 1 + 1 + 5 * TINY.shape.n_layers + 1 + 1


def test_measured_traffic_follows_the_profile_hash(tmp_path, monkeypatch):
    v = bench.measured_traffic("k_chain(o+gate_up+down+next_qkv)")
    recorded = re.search(r"dram bytes per launch \(M = 1\): (\d+)",
                         open(os.path.join(REPO, "profiles", "k_chain_llama2-7b.md")).read())
    assert v is None or v == int(recorded.group(1))
    assert v is None or 4.0e8 < v < 4.3e8  # one launch's weights (401.6 MB) plus a little
    assert bench.measured_traffic("k_attn") is None  # no traffic summary for it
    # a profile whose recorded hash differs from the sources gives no number
    prof = tmp_path / "profiles"
    prof.mkdir()
    text = open(os.path.join(REPO, "profiles", "k_chain_llama2-7b.md")).read()
    digest = re.search(r"`([0-9a-f]{64})`", text).group(1)
    other = ("0" if digest[0] != "0" else "1") + digest[1:]
    (prof / "k_chain_llama2-7b.md").write_text(text.replace(digest, other))
    csrc = tmp_path / "paper_2606_03113_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for f in bench.TRAFFIC_SOURCES:
        (csrc / f).write_bytes(open(os.path.join(REPO, "paper_2606_03113_gb300", "csrc", f),
                                    "rb").read())
    monkeypatch.setattr(bench, "REPO", str(tmp_path))
    assert bench.measured_traffic("k_chain(o+gate_up+down+next_qkv)") is None


def test_clock_record_parser(tmp_path):
    path = tmp_path / "clocks.csv"
    rows = ["0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active",
            "0, 2055, 2070, 950.0, 0x4, Not Active, Not Active, Not Active, Active",
            "0, 2070, 2070, 960.0, 0x0, Not Active, Not Active, Not Active, Not Active",
            "garbage line"]
    path.write_text("\n".join(rows) + "\n")
    cs = bench.ClockSampler(0)
    cs.path = str(path)
    out = cs.summary()
    assert out["sm_mhz"] == 2070.0 and out["sm_max_mhz"] == 2070.0
    assert out["reasons"] == ["sw_power_cap"] and out["samples"] == 3
    assert not path.exists()  # the record is removed after reading


def test_reference_arm_prints_the_contract_line():
    """`bench.py --impl reference` times the oracle on the host cores and
    prints one JSON line with the contract's keys (tiny workload here)."""
    import json
    import subprocess
    out = subprocess.check_output(
        [sys.executable, os.path.join(REPO, "bench.py"), "--impl", "reference", "--workload",
         "tiny", "--steps", "1", "--warmup", "0"], text=True, timeout=300, cwd=REPO)
    lines = [l for l in out.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config"):
        assert key in d, key
    assert d["impl"] == "reference" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == dict(value=d["value"], unit=d["unit"], h2d_bytes_per_step=0,
                            d2h_bytes_per_step=0)


def test_static_grid_sweeps_every_point_and_keeps_the_best(monkeypatch):
    """compare.static_best: every candidate exit layer x every draft length
    is timed on the short generation, the three fastest are timed again on
    the full one, and the best of those is reported with its settings."""
    from dataclasses import replace
    w = replace(LLAMA2_7B, candidates=(4, 8, 12), kmax=3)
    calls = []
    speed = {(4, 1): 50.0, (8, 2): 90.0, (8, 3): 80.0, (12, 1): 85.0}
    state = {}

    def set_policy(kind, l=0, k=0, **_):
        assert kind == "static"
        state["lk"] = (l, k)

    def fake_time_generate(eng, ids, n_new, barrier):
        l, k = state["lk"]
        calls.append((l, k, n_new))
        tok_s = speed.get((l, k), 10.0) * (0.9 if n_new == 256 and (l, k) == (8, 2) else 1.0)
        trace = [dict(pos=600, kcap=k, visited=[l], lstar=l, k=k, a=k)]
        return 1e3 * n_new / tok_s, n_new, trace

    monkeypatch.setattr(bench, "time_generate", fake_time_generate)
    best = bench.static_grid(w, set_policy, None, [0] * 8, 256, lambda: None, n_grid=64, top=3)
    timed = {(l, k) for l, k, n in calls if n == 64}
    assert timed == {(l, k) for l in (4, 8, 12) for k in (1, 2, 3)}
    again = [(l, k) for l, k, n in calls if n == 256]
    assert sorted(set(again)) == [(8, 2), (8, 3), (12, 1)]  # the three fastest short runs
    # (8, 2) is fastest on 64 tokens but slower on the full run: (12, 1) wins
    assert (best["l"], best["k"]) == (12, 1) and best["tok_s"] == pytest.approx(85.0)
    assert best["grid_top"][0] == dict(l=8, k=2, tok_s=90.0)
