"""The ncu recipes under profiles/ follow the profiling rules of this project: every
ncu command leaves the GPU clocks alone (--clock-control none), and every capture
that collects more than launch times (a section set or sections) names one kernel
(-k) and at most three launches (-c)."""
import glob
import os
import re
import shlex

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _code_commands(path):
    """Shell commands in the fenced code blocks of one file: continuation lines
    joined, NAME="..." assignments substituted into the lines after them."""
    cmds, env, fenced, buf = [], {}, False, ""
    for raw in open(path, encoding="utf-8"):
        line = raw.rstrip("\n")
        if line.lstrip().startswith("```"):
            fenced, buf = not fenced, ""
            continue
        if not fenced:
            continue
        if line.endswith("\\"):
            buf += line[:-1] + " "
            continue
        line, buf = buf + line, ""
        m = re.fullmatch(r'\s*([A-Z][A-Z0-9_]*)="(.*)"\s*', line)
        if m:
            env[m.group(1)] = re.sub(r"\$([A-Z][A-Z0-9_]*)", lambda v: env.get(v.group(1), v.group(0)), m.group(2))
            continue
        cmds.append(re.sub(r"\$([A-Z][A-Z0-9_]*)", lambda v: env.get(v.group(1), v.group(0)), line))
    return cmds


def _ncu_commands():
    out = []
    for path in sorted(glob.glob(os.path.join(ROOT, "profiles", "*.md"))):
        for cmd in _code_commands(path):
            if re.match(r"\s*ncu\s", cmd):
                out.append((os.path.basename(path), cmd))
    return out


def test_profiles_hold_ncu_recipes():
    assert len(_ncu_commands()) >= 5


def test_every_ncu_recipe_leaves_the_clocks_alone():
    for name, cmd in _ncu_commands():
        argv = shlex.split(cmd)
        i = argv.index("--clock-control") if "--clock-control" in argv else -1
        assert i >= 0 and argv[i + 1] == "none", f"{name}: {cmd}"


def test_section_captures_name_one_kernel_and_few_launches():
    for name, cmd in _ncu_commands():
        argv = shlex.split(cmd)
        if "--set" not in argv and "--section" not in argv:
            continue
        assert "-k" in argv, f"{name}: a section capture without -k: {cmd}"
        assert "-c" in argv and int(argv[argv.index("-c") + 1]) <= 3, f"{name}: {cmd}"
