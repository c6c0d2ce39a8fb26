"""bench.py's reference arm (the CPU oracle) and its launch contract, on CPU.

The reference arm needs no GPU: it times the oracle on this host's cores and
prints one JSON line with the keys the driver reads. Under a multi-rank launch
only rank 0 runs it; every other rank exits 0 without work or output.
"""
from __future__ import annotations

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ARGS = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "1",
        "--steps", "1", "--warmup", "0"]


def _run(extra_env: dict, extra_args: tuple = ()) -> subprocess.CompletedProcess:
    env = dict(os.environ)
    env.update(extra_env)
    return subprocess.run(ARGS + list(extra_args), cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)


def test_reference_arm_prints_one_line():
    r = _run({"RANK": "0", "WORLD_SIZE": "1"})
    assert r.returncode == 0, r.stderr
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference"
    assert line["unit"] == "pairs/s" and line["higher_is_better"] is True
    assert line["config"]["workload"] == "tools-K100-V32000-B1-f32"
    assert line["config"]["N_nodes"] == 1384
    # the GPU arm prints the same config object (bench.workload_config), so the
    # two arms' lines describe one workload key for key
    sys.path.insert(0, ROOT)
    import bench
    from paper_2608_12574_gb300 import workloads as W
    assert line["config"] == bench.workload_config(W.config(1), 1384)
    assert set(line["config"]) == {"workload", "K", "V", "batch", "decode_steps", "N_nodes", "N_chars", "r", "l2"}
    assert line["value"] > 0 and line["steps"] == 1 and line["warmup"] == 0
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"]
    assert cb["value"] == line["value"]
    e2e = line["e2e"]
    assert e2e == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}
    # pairs/s of the sample: the sampled share of N x V pairs over one step's time
    assert line["ms_per_step"] > 0
    pairs = line["value"] * line["ms_per_step"] * 1e-3
    assert abs(pairs - 1384 * 32000 * _share(cb)) <= 1e-3 * pairs   # the share is printed to 4 digits


def _share(cb: dict) -> float:
    # "... a 0.7756 slice of one ... step: 1074 of 1384 mask rows ..."
    words = cb["sample"].split()
    return float(words[words.index("slice") - 1]) if "slice" in words else float("nan")


def test_reference_arm_other_ranks_exit_quietly():
    r = _run({"RANK": "1", "WORLD_SIZE": "2"}, ("--gpus", "2"))
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == ""


def test_gpus_must_match_the_launch():
    """A launch of WORLD_SIZE ranks whose --gpus says otherwise fails loudly
    instead of reporting a different number of GPUs."""
    r = _run({"RANK": "0", "WORLD_SIZE": "2"}, ("--gpus", "4"))
    assert r.returncode != 0
    assert "does not match WORLD_SIZE" in r.stderr


def test_clock_summary_parses_nvidia_smi_samples():
    """The clock record of the timed region: median SM clock, the maximum, and
    every throttle reason seen Active in any sample (sw_power_cap included)."""
    sys.path.insert(0, ROOT)
    import bench
    c = bench.ClockSampler(None)
    c.out = "\n".join([
        "2070, 2070, 812.4, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "1980, 2070, 1391.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "2055, 2070, 1102.7, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "[N/A], [N/A], [N/A], [N/A], [N/A], [N/A], [N/A], [N/A]",
        "garbage",
    ])
    s = c.summary()
    assert s == {"sm_mhz": 2055.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}
    c.out = "1200, 2070, 900.0, 0x0000000000000008, Active, Not Active, Active, Not Active"
    assert c.summary()["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]
    c.out = ""
    assert c.summary()["reasons"] == ["no samples"]


def test_kernel_source_hash_ignores_comments_only(tmp_path):
    import bench
    a, b, c = tmp_path / "a.cu", tmp_path / "b.cu", tmp_path / "c.cu"
    a.write_text("// header\nint f() { return 1; }  // one\n\n")
    b.write_text("// another header\n\nint f() { return 1; }\n// trailing\n")
    c.write_text("int f() { return 2; }\n")
    assert bench.kernel_source_hash(str(a)) == bench.kernel_source_hash(str(b))
    assert bench.kernel_source_hash(str(a)) != bench.kernel_source_hash(str(c))


def test_compile_kernels_follows_the_library_rule():
    """gpu_launches counts 2 compile kernels (fill, then the pair search ORing
    its hits) only for masks of at most 32 MB, tries of at most 128 nodes per
    SM, tokens and depth within 16 bytes and no repeated token string; else 3."""
    import types
    import bench
    from paper_2608_12574_gb300 import workloads as W

    def vocab(strings):
        vb, vo = W.pack(list(strings) + [b""])  # the last token is EOS
        return types.SimpleNamespace(vocab_bytes=vb, vocab_offsets=vo, V=len(strings) + 1)

    small = vocab([bytes([97 + i % 26]) * (1 + i % 5) + str(i).encode() for i in range(1000)])
    assert bench.compile_kernels(small, 1384, 20, 152) == 2
    assert bench.compile_kernels(small, 152 * 128 + 1, 20, 152) == 3          # too many nodes for two lanes each
    assert bench.compile_kernels(small, 152 * 128, 20, 152) == 2
    assert bench.compile_kernels(vocab([b"x" * 17, b"a"]), 100, 20, 152) == 3  # a token longer than 16 bytes
    assert bench.compile_kernels(vocab([b"x" * 17, b"a"]), 100, 16, 152) == 2  # ... that no path of the trie reaches
    assert bench.compile_kernels(vocab([b"ab", b"cd", b"ab"]), 100, 20, 152) == 3  # a repeated token string
    wide = vocab([str(i).encode() for i in range(300000)])   # V = 300,001: 9,376 words, 37,504 B per row
    assert bench.compile_kernels(wide, 894, 20, 152) == 2     # 33,528,576 B <= 32 MB
    assert bench.compile_kernels(wide, 895, 20, 152) == 3     # 33,566,080 B > 32 MB
