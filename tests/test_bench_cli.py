"""bench.py's command surface on the CPU: every `--sweep` choice has its sweep function,
and every library function bench.py calls exists in the Python binding (a renamed hook
would otherwise fail only on the GPU, minutes into a run)."""
import os
import re
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    sys.path.insert(0, ROOT)
    import bench
    return bench


def test_every_sweep_choice_has_its_function():
    bench = _bench()
    src = open(os.path.join(ROOT, "bench.py")).read()
    choices = re.search(r'"--sweep", choices=\[([^\]]*)\]', src).group(1)
    for name in re.findall(r'"(\w+)"', choices):
        assert callable(getattr(bench, f"run_{name}_sweep", None)), f"--sweep {name}: run_{name}_sweep missing"


def test_every_library_call_exists_in_the_binding():
    import paper_2609_29219_gb300 as m
    src = open(os.path.join(ROOT, "bench.py")).read()
    called = set(re.findall(r"\bloom\.(loom_\w+)\(", src))
    assert called, "bench.py calls the library through `loom.`"
    missing = sorted(n for n in called if not hasattr(m, n))
    assert not missing, f"bench.py calls functions the binding does not have: {missing}"
