"""The committed ncu summaries under profiles/: each names the command that
made it (an ncu run of committed files with --clock-control none), and the
summaries the benchmark reads DRAM traffic from carry a numeric figure
(CPU only)."""
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PROF = os.path.join(ROOT, "profiles")


def _profiles():
    return sorted(f for f in os.listdir(PROF) if f.endswith(".md"))


@pytest.mark.parametrize("name", _profiles())
def test_profile_names_its_command(name):
    text = open(os.path.join(PROF, name)).read()
    if name == "measured_roofs.md":
        assert "python bench.py" in text
        return
    cmds = [ln.strip() for ln in text.splitlines() if ln.strip().startswith("ncu ")]
    assert cmds, f"{name}: no ncu command"
    for c in cmds:
        assert "--clock-control none" in c, f"{name}: {c}"
    # the command runs committed files only
    assert "_work/" not in text, name


@pytest.mark.parametrize("kernel,key", [
    ("ppo_persistent_kernel", "traffic_bytes_per_launch"),
    ("fleet_windows_kernel", "traffic_bytes_per_launch"),
    ("mlp_bf16_pair_kernel", "traffic_bytes_per_launch"),
    ("gae_stream_kernel", "traffic_bytes_per_env_step_v1"),
    ("gae_stream_kernel", "traffic_bytes_per_env_step_v4"),
])
def test_bench_traffic_figures(kernel, key):
    """bench.py reads these keys (bench.load_traffic / load_traffic_per_unit)."""
    text = open(os.path.join(PROF, kernel + ".md")).read()
    m = re.search(r"^" + re.escape(key) + r":\s*([0-9.]+)\s*$", text, re.M)
    assert m, f"{kernel}.md lacks {key}"
    assert float(m.group(1)) > 0
