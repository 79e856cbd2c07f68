"""Planted mistakes in the oracle, on the CPU: do the pins catch them?

Each mutant below is one plausible error in one step of the oracle: a bridge off by one, a
dropped 1/sqrt(d), K and V swapped, an interleaved GQA map, a dropped term of the softmax
gradient, a shifted ring slot, and so on. For each, a copy of ``oracle/pbb_oracle.c`` with that
single change is compiled in a temporary directory. Every pin of ``tests/test_oracle.py`` then
runs against it in a child process, so that a mutant that corrupts memory cannot take the test
run down, and at least one pin must fail. The unchanged source, under the same harness, must
pass them all.

Run as a script (``python tests/test_oracle_mutants.py SRC BUILD_DIR``) it is that child
process: exit 0 if every pin passes against the oracle built from SRC, 1 at the first failure,
2 if SRC does not compile (which must not pass for a caught mutant).
"""
from __future__ import annotations

import concurrent.futures
import importlib.util
import itertools
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
ORACLE_SRC = os.path.join(ROOT, "oracle", "pbb_oracle.c")
ORACLE_INIT = os.path.join(ROOT, "oracle", "__init__.py")
PINS = os.path.join(HERE, "test_oracle.py")

# (name, text in pbb_oracle.c, replacement): each text occurs exactly once in the source.
MUTANTS = [
    ("bridge one position short", "s >= p - h && s <= p - 1", "s >= p - h + 1 && s <= p - 1"),
    ("bridge kept one step too long", "r < h && s >= p - h", "r <= h && s >= p - h"),
    ("block prefix drops its first position", "if (s >= p) return 1;", "if (s > p) return 1;"),
    ("softmax without 1/sqrt(d)", "const double scale = 1.0 / sqrt((double)d);\n    double m = -INFINITY;",
     "const double scale = 1.0;\n    double m = -INFINITY;"),
    ("forward reads K and V swapped", "kr[m] = k + (head + (size_t)s) * d;\n                vr[m] = v + (head + (size_t)s) * d;",
     "kr[m] = v + (head + (size_t)s) * d;\n                vr[m] = k + (head + (size_t)s) * d;"),
    ("forward with interleaved GQA heads", "const long kv = j / group;", "const long kv = j % Hkv;"),
    ("log-partition in base 2", "*lse = m + log(den)", "*lse = m + log2(den)"),
    ("softmax gradient without its row term", "const double dz = P[i] * (dP[i] - sum_pdp);",
     "const double dz = P[i] * dP[i];"),
    ("dq without 1/sqrt(d)", "dqt[c] += dz * ks[c] * scale;", "dqt[c] += dz * ks[c];"),
    ("dv from the score gradient", "dvs[c] += P[i] * dot_[c];", "dvs[c] += dz * dot_[c];"),
    ("dk with the wrong sign", "dks[c] += dz * qt[c] * scale;", "dks[c] -= dz * qt[c] * scale;"),
    ("dk from k instead of q", "dks[c] += dz * qt[c] * scale;", "dks[c] += dz * ks[c] * scale;"),
    ("backward without 1/sqrt(d)", "const double scale = 1.0 / sqrt((double)d);\n    memset(dq",
     "const double scale = 1.0;\n    memset(dq"),
    ("window one position wide", "s >= t - w + 1;", "s >= t - w;"),
    ("ring slot shifted by one", "const long slot = t[bi] % b;", "const long slot = (t[bi] + 1) % b;"),
    ("ring interval starts one late", "long a = h * (tb / h - 1);", "long a = h * (tb / h - 1) + 1;"),
    ("bf16 widened from the low half", "(uint32_t)h << 16", "(uint32_t)h"),
]


def _load_module(name: str, path: str):
    spec = importlib.util.spec_from_file_location(name, path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _pin_calls(pins):
    """Every (test name, function, kwargs) of the pin module, parametrisations expanded."""
    for name in sorted(n for n in dir(pins) if n.startswith("test_")):
        fn = getattr(pins, name)
        axes = []
        for mark in getattr(fn, "pytestmark", []):
            if mark.name != "parametrize":
                continue
            names = [a.strip() for a in mark.args[0].split(",")]
            values = [v if len(names) > 1 else (v,) for v in mark.args[1]]
            axes.append([dict(zip(names, v)) for v in values])
        for combo in itertools.product(*axes) if axes else [()]:
            kwargs = {}
            for part in combo:
                kwargs.update(part)
            yield name, fn, kwargs


def run_pins(src: str, build_dir: str) -> int:
    """Build the oracle from `src` into `build_dir` and run every pin; 0 if all pass."""
    oracle = _load_module("oracle_under_test", ORACLE_INIT)
    oracle._SRC = src
    oracle._BUILD = build_dir
    oracle._LIB_PATH = os.path.join(build_dir, "liboracle.so")
    oracle._lib = None
    try:
        oracle.build()
    except Exception as e:  # noqa: BLE001
        print(f"build failed: {e}")
        return 2
    pins = _load_module("oracle_pins", PINS)
    for name, fn, kwargs in _pin_calls(pins):
        try:
            fn(oracle, **kwargs)
        except Exception as e:  # noqa: BLE001 - any failure of a pin counts
            print(f"pin failed: {name} {kwargs}: {type(e).__name__}: {str(e)[:200]}")
            return 1
    print("all pins pass")
    return 0


def _child(src: str, build_dir: str):
    env = dict(os.environ, OMP_NUM_THREADS="2")
    return subprocess.run([sys.executable, os.path.abspath(__file__), src, build_dir], capture_output=True,
                          text=True, timeout=600, env=env, cwd=ROOT)


def test_pins_catch_every_planted_mistake(tmp_path):
    source = open(ORACLE_SRC).read()
    jobs = [("unchanged", source)]
    for name, old, new in MUTANTS:
        assert source.count(old) == 1, f"mutant '{name}': its text must occur once in the oracle"
        jobs.append((name, source.replace(old, new)))
    args = []
    for i, (name, text) in enumerate(jobs):
        d = tmp_path / f"m{i}"
        d.mkdir()
        (d / "pbb_oracle.c").write_text(text)
        args.append((name, str(d / "pbb_oracle.c"), str(d)))
    workers = max(1, min(8, (os.cpu_count() or 2) // 2))
    with concurrent.futures.ThreadPoolExecutor(max_workers=workers) as ex:
        results = list(ex.map(lambda a: (a[0], _child(a[1], a[2])), args))
    control = results[0][1]
    assert control.returncode == 0, "the unchanged oracle must pass every pin:\n" + control.stdout + control.stderr
    unbuilt = [name for name, r in results[1:] if r.returncode == 2]
    assert not unbuilt, f"mutants that do not compile: {unbuilt}"
    survivors = [name for name, r in results[1:] if r.returncode == 0]
    assert not survivors, f"mutants no pin catches: {survivors}"
    for name, r in results[1:]:
        assert r.returncode == 1 and "pin failed" in r.stdout, f"mutant '{name}' ended unexpectedly:\n{r.stdout}{r.stderr}"


if __name__ == "__main__":
    sys.path.insert(0, ROOT)
    sys.path.insert(0, HERE)
    sys.exit(run_pins(sys.argv[1], sys.argv[2]))
