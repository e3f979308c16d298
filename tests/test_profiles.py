"""The committed ncu summaries: every one names the command that made it
(committed files only), and the benchmark takes its DRAM-traffic figure from
a summary only while that summary's kernel source is the current one."""
import glob
import hashlib
import os
import re

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PROFILES = sorted(glob.glob(os.path.join(ROOT, "profiles", "*.md")))


def _fields(path):
    return dict(line.split(": ", 1) for line in open(path).read().splitlines()
                if re.match(r"^[a-z_0-9]+: ", line))


def test_every_summary_has_its_command_and_no_working_files():
    assert PROFILES
    for p in PROFILES:
        text = open(p).read()
        assert "```" in text and ("ncu " in text or "python bench.py" in text), p
        assert "_work" not in text, p
        # every python script named in a command is a committed file
        for script in re.findall(r"python ([\w/]+\.py)", text):
            assert os.path.exists(os.path.join(ROOT, script)), (p, script)


def test_traffic_ratio_follows_the_kernel_source():
    path = os.path.join(ROOT, "profiles", "attend_kernel_long_context_32k_int2.md")
    f = _fields(path)
    sha = hashlib.sha256(open(os.path.join(ROOT, "paper_2609_32831_gb300", "csrc", "attend.cu"), "rb")
                         .read()).hexdigest()[:16]
    got = bench.profiled_traffic_ratio()
    if f["source_sha256_16"].strip() == sha:
        assert got == float(f["traffic_ratio"])
        # DRAM traffic close to the algorithmic bytes: no re-reads
        assert 1.0 <= got < 1.1
    else:
        assert got is None
