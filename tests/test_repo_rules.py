"""Rules of the repository that can be checked by reading it (no GPU): the product package
never reaches the oracle, and every committed profile gives a runnable ncu command that leaves
the GPU clocks alone."""
import glob
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_product_package_does_not_use_the_oracle():
    pkg = os.path.join(ROOT, "paper_2606_12876_gb300")
    files = glob.glob(os.path.join(pkg, "*.py")) + glob.glob(os.path.join(pkg, "csrc", "*"))
    assert files
    for f in files:
        text = open(f, errors="replace").read()
        assert not re.search(r"^\s*(import|from)\s+oracle\b", text, re.M), f
        assert "liboracle" not in text and "oracle_" not in text, f


def test_profiles_give_ncu_commands_with_clock_control_off():
    docs = glob.glob(os.path.join(ROOT, "profiles", "*.md"))
    assert docs
    for f in docs:
        text = open(f).read()
        lines = [l for l in text.splitlines() if re.search(r"^\s*ncu\s", l)]
        assert lines, "%s: no ncu command" % f
        for l in lines:
            assert "--clock-control none" in l, (f, l)
        assert "_work" not in text, f
