"""The committed ncu summaries: each gives the command that made it, with
`--clock-control none` (ncu otherwise locks the GPU's clocks), running only
committed files; each row-pass summary carries the source hash and the
per-launch traffic that bench.py reads, and that traffic is within 1% of the
algorithmic bytes the summary states, plus the top-k lists a filtered pass
writes (a capture that re-read the logits would show more)."""
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SUMMARIES = sorted(glob.glob(os.path.join(ROOT, "profiles", "*")))


def _command(text):
    # the indented block that starts with ncu, joined across continuation lines
    lines = text.splitlines()
    for i, line in enumerate(lines):
        if line.strip().startswith("ncu "):
            cmd = []
            for l in lines[i:]:
                cmd.append(l.strip().rstrip("\\").strip())
                if not l.rstrip().endswith("\\"):
                    break
            return " ".join(cmd)
    return None


def test_profiles_hold_only_short_text():
    assert SUMMARIES
    for path in SUMMARIES:
        assert os.path.splitext(path)[1] in (".md", ".txt"), path
        assert os.path.getsize(path) < 16 * 1024, path


@pytest.mark.parametrize("path", SUMMARIES, ids=os.path.basename)
def test_each_summary_gives_its_command(path):
    cmd = _command(open(path).read())
    assert cmd is not None, path
    assert "--clock-control none" in cmd
    assert " python bench.py" in cmd  # the committed benchmark, nothing else
    assert "_work" not in cmd and "/root" not in cmd


@pytest.mark.parametrize("path", [p for p in SUMMARIES
                                  if os.path.basename(p).startswith("rowpass_")],
                         ids=os.path.basename)
def test_row_pass_summaries_carry_hash_and_traffic(path):
    text = open(path).read()
    assert re.search(r"^- source_sha256: `[0-9a-f]{16}`$", text, re.M), path
    m = re.search(r"^- traffic_bytes_per_launch: (\d+)$", text, re.M)
    assert m, path
    traffic = int(m.group(1))
    # the algorithmic bytes of a full launch: the scaled figure when the
    # capture was a cut of the workload, else the captured launch's
    full = re.search(r"x ([\d,]+) / ([\d,]+) = ([\d,]+) bytes", text)
    if full:
        algo = int(full.group(1).replace(",", ""))
        assert int(full.group(3).replace(",", "")) == traffic
    else:
        algo = int(re.search(r"Algorithmic bytes per launch: ([\d,]+)", text)
                   .group(1).replace(",", ""))
    # with filters the pass also writes top_k entries of 8 bytes per 8 KB unit
    k = re.search(r"^- top_k: (\d+)$", text, re.M)
    lists = int(k.group(1)) * 8 / 8192 if k else 0.0
    assert algo <= traffic <= (1.01 + lists) * algo + 16e6, (traffic, algo)
