"""The committed ncu summaries: each gives the command that made it, the command
runs committed files only and never lets ncu lock the clocks, and every
per-kernel traffic entry the bench reads names a source file and workload that
exist."""
import json
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PROFILES = os.path.join(ROOT, "profiles")
CSRC = os.path.join(ROOT, "paper_2609_27233_gb300", "csrc")


def summaries():
    return sorted(f for f in os.listdir(PROFILES) if f.endswith(".md"))


def test_every_summary_gives_its_ncu_command_with_clock_control_none():
    assert summaries()
    for f in summaries():
        text = open(os.path.join(PROFILES, f)).read()
        cmds = re.findall(r"```\n(.*?)```", text, flags=re.S)
        assert cmds, f"{f}: no command block"
        joined = "\n".join(cmds)
        assert "ncu " in joined, f
        for line in re.findall(r"ncu (?:[^\n]*\\\n)*[^\n]*", joined):   # continued lines included
            assert "--clock-control none" in line, (f, line)


def test_summary_commands_run_committed_files_only():
    for f in summaries():
        text = open(os.path.join(PROFILES, f)).read()
        for block in re.findall(r"```\n(.*?)```", text, flags=re.S):
            assert "_work/" not in block and "gpurun" not in block, f
            for script in re.findall(r"python ([\w/]+\.py)", block):
                assert os.path.exists(os.path.join(ROOT, script)), (f, script)


def test_profiles_hold_text_only():
    for f in os.listdir(PROFILES):
        assert f.endswith((".md", ".txt", ".json")), f
        assert os.path.getsize(os.path.join(PROFILES, f)) < 64 * 1024, f


def test_traffic_entries_name_existing_sources_and_bench_workloads():
    prof = json.load(open(os.path.join(PROFILES, "ncu_traffic.json")))
    bench = open(os.path.join(ROOT, "bench.py")).read()
    workloads = set(re.search(r'choices=\["llama8b_layer",[^\]]*\]', bench).group(0)[9:-1].replace('"', "")
                    .replace(" ", "").replace("\n", "").split(","))
    assert prof
    for label, e in prof.items():
        assert os.path.exists(os.path.join(CSRC, e["source"])), label
        assert re.fullmatch(r"[0-9a-f]{16}", e["source_sha"]), label
        assert e["workload"] in workloads, (label, e["workload"])
        assert e["bytes_per_launch_full"] == e["dram_read"] + e["dram_write"], label
        assert "--clock-control none" in e["capture"] and "ncu " in e["capture"], label
