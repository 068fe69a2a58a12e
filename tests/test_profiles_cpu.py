"""The committed ncu summaries: each gives the command that made it, every
profiling command leaves the GPU clocks alone, and each runs committed files
only (the benchmark at the repository root)."""
import os
import re

import pytest

REPO = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PROFILES = os.path.join(REPO, "profiles")
NAMES = sorted(f for f in os.listdir(PROFILES) if f.endswith((".md", ".txt")))


def _commands(text):
    """Indented command lines (the summaries' code blocks), joined across
    trailing backslashes."""
    out, cur = [], ""
    for line in text.splitlines():
        if not line.startswith("    "):
            continue
        cur += " " + line.strip()
        if cur.endswith("\\"):
            cur = cur[:-1]
            continue
        out.append(cur.strip())
        cur = ""
    return out


def test_there_are_summaries():
    assert NAMES


@pytest.mark.parametrize("name", NAMES)
def test_summary_names_its_command(name):
    text = open(os.path.join(PROFILES, name)).read()
    assert re.search(r"^Command", text, re.M), name
    cmds = _commands(text)
    profiling = [c for c in cmds if c.startswith("ncu ") and " -i " not in c]
    assert profiling, name
    for c in profiling:
        # ncu locks the clocks unless told not to
        assert "--clock-control none" in c, (name, c)
        # the profiled program is the committed benchmark
        assert "python bench.py" in c, (name, c)
    for c in cmds:
        assert "_work" not in c, (name, c)
        if c.startswith("python "):
            script = c.split()[1]
            assert os.path.isfile(os.path.join(REPO, script)), (name, script)


@pytest.mark.parametrize("name", NAMES)
def test_summary_is_short_text(name):
    assert os.path.getsize(os.path.join(PROFILES, name)) < 16 * 1024, name
