"""The ncu summaries under profiles/: every ncu command they give leaves the
GPU clocks alone, and every command runs committed files only."""
from __future__ import annotations

import os
import re
import subprocess

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PROFILES = os.path.join(ROOT, "profiles")


def _summaries():
    return [os.path.join(PROFILES, f) for f in sorted(os.listdir(PROFILES)) if f.endswith(".md")]


def _commands(text):
    """Indented command blocks (four spaces), joined across continuation lines."""
    cmds, cur = [], []
    for line in text.splitlines():
        if line.startswith("    ") and line.strip():
            cur.append(line.strip().rstrip("\\").strip())
        elif cur:
            cmds.append(" ".join(cur))
            cur = []
    if cur:
        cmds.append(" ".join(cur))
    return cmds


def test_every_ncu_command_keeps_the_clocks():
    for path in _summaries():
        for cmd in _commands(open(path).read()):
            if re.search(r"(^|\s|&&\s*)ncu\s", cmd):
                assert "--clock-control none" in cmd, (os.path.basename(path), cmd)


def test_commands_run_committed_files_only():
    tracked = set(subprocess.run(["git", "ls-files"], cwd=ROOT, capture_output=True, text=True).stdout.split())
    if not tracked:
        return                                   # not a git checkout
    for path in _summaries():
        for cmd in _commands(open(path).read()):
            assert "_work" not in cmd, (os.path.basename(path), cmd)
            for script in re.findall(r"python\s+(?:-m\s+)?([\w./-]+\.py)", cmd):
                assert script in tracked, (os.path.basename(path), script)
            for mod in re.findall(r"python\s+-m\s+([\w.]+)(?:\s|$)", cmd):
                if mod in ("pytest",):
                    continue
                rel = mod.replace(".", "/")
                assert f"{rel}.py" in tracked or f"{rel}/__init__.py" in tracked, (os.path.basename(path), mod)
