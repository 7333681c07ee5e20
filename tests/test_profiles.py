"""The summaries under profiles/ give the commands that produced their figures.
Every `kernel_bench` and `bench.py` invocation in them must parse with the
current committed parsers, so that the commands run committed files only.
No GPU."""
import glob
import os
import re
import shlex
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _commands():
    out = []
    for path in sorted(glob.glob(os.path.join(ROOT, "profiles", "*.md"))):
        text = open(path).read()
        for block in re.findall(r"```\n(.*?)```", text, flags=re.S):
            cmd = block.replace("\\\n", " ")
            for line in cmd.splitlines():
                if "kernel_bench" in line or "bench.py" in line:
                    out.append((os.path.basename(path), line.strip()))
    return out


CMDS = _commands()


def test_profiles_have_commands():
    names = {n for n, _ in CMDS}
    for path in glob.glob(os.path.join(ROOT, "profiles", "*.md")):
        assert os.path.basename(path) in names, f"{path} gives no command"


@pytest.mark.parametrize("name,line", CMDS)
def test_profile_command_parses(name, line, monkeypatch):
    toks = shlex.split(line)
    if "paper_2608_02474_gb300.kernel_bench" in toks:
        from paper_2608_02474_gb300 import kernel_bench
        kernel_bench.make_parser().parse_args(
            toks[toks.index("paper_2608_02474_gb300.kernel_bench") + 1:])   # exits on a bad option
    else:
        script = [t for t in toks if t.endswith("bench.py")][0]
        args = toks[toks.index(script) + 1:]
        import bench
        monkeypatch.setattr(sys, "argv", ["bench.py"] + args)
        bench.parse()   # exits on an unknown option
