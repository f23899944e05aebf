"""Planted mistakes: the pins must catch a plausible error in the oracle.

Each case copies the oracle's source, plants one mistake of the kinds a
transcription of the method could make (a wrong sign, a dropped term, a wrong
index or tie rule, a transposed operand, a wrong normalisation or order),
builds or loads the copy on the CPU and runs the pins of
``test_oracle_pins.py`` / ``test_oracle_pca_pins.py`` against it.  At least one
pin has to fail.  The oracle itself is untouched: the copies live in pytest's
temporary directory and are swapped in only for the duration of a case.  Every
planted C mistake keeps all memory accesses in bounds.
"""
import os
import shutil
import subprocess
import types

import pytest

import oracle
from tests import test_oracle_pca_pins as pca_pins
from tests import test_oracle_pins as pins

ORACLE_DIR = os.path.dirname(os.path.abspath(oracle.__file__))

# (what, original snippet, planted snippet); each snippet occurs once in oracle.c
C_MUTANTS = [
    ("assign: x + c instead of x - c",
     "double t = feat(X, dtype, ldx, i, j) - Ct[k * d + j];",
     "double t = feat(X, dtype, ldx, i, j) + Ct[k * d + j];"),
    ("assign: the last dimension dropped",
     "        for (int64_t k = 0; k < K; ++k) {\n            double s = 0.0;\n            for (int64_t j = 0; j < d; ++j) {",
     "        for (int64_t k = 0; k < K; ++k) {\n            double s = 0.0;\n            for (int64_t j = 0; j < d - 1; ++j) {"),
    ("assign: ties to the highest index",
     "            if (s < best) {",
     "            if (s <= best) {"),
    ("assign: the centre table read transposed",
     "- Ct[k * d + j];",
     "- Ct[j * K + k];"),
    ("assign: runner-up not kept when the best moves",
     "                second = best;\n",
     ""),
    ("update: mean divided by n + 1",
     "(float)(sums[k * d + j] / (double)counts[k]);",
     "(float)(sums[k * d + j] / (double)(counts[k] + 1));"),
    ("update: re-seed takes the nearest point",
     "mi > (mind ? mind[far] : 0.0)",
     "mi < (mind ? mind[far] : 0.0)"),
    ("update: a re-seed point may be used twice",
     "        used[far] = 1;\n",
     ""),
    ("partition: buckets filled in descending index",
     "    for (int64_t i = 0; i < N; ++i) {\n        int64_t s = fill[labels[i]]++;",
     "    for (int64_t i = N - 1; i >= 0; --i) {\n        int64_t s = fill[labels[i]]++;"),
    ("k-means++: D^2 against the newest centre only",
     "            if (k == 0 || dj < D2[j])",
     "            if (1)"),
    ("k-means++: sampling proportional to D instead of D^2",
     "                D2[j] = dj;",
     "                D2[j] = sqrt(dj);"),
    ("bf16: truncation instead of round-to-nearest-even",
     "    u += 0x7FFFu + lsb;",
     "    u += 0u * lsb;"),
    ("splitmix64: the counter starts at 0",
     "uint64_t z = seed + (j + 1) * SM64_GAMMA;",
     "uint64_t z = seed + j * SM64_GAMMA;"),
    ("objective: the centre table indexed without its row stride",
     "- Ct[(int64_t)labels[i] * d + j];",
     "- Ct[(int64_t)labels[i] + j];"),
    ("objective: unsquared distances summed",
     "        J += s;\n    }\n    free(Ct);\n    *objective = J;",
     "        J += sqrt(s);\n    }\n    free(Ct);\n    *objective = J;"),
    ("tag statistics: l1 / l2^2 instead of l1 / l2",
     "l1 / sqrt(l2sq)",
     "l1 / l2sq"),
]

# (what, original snippet, planted snippet); each snippet occurs once in pca.py
PCA_MUTANTS = [
    ("covariance about the origin (no centring)", "    Y = X64 - mu\n", "    Y = X64\n"),
    ("covariance normalised by N - 1", "(Y.T @ Y) / X64.shape[0]", "(Y.T @ Y) / (X64.shape[0] - 1)"),
    ("eigenvectors read as rows", "vecs[:, order[:r]].T", "vecs[order[:r], :]"),
    ("components in increasing variance", "np.argsort(-vals, kind=\"stable\")", "np.argsort(vals, kind=\"stable\")"),
    ("projection without centring",
     "(X64 - np.asarray(mu, dtype=np.float64)) @", "X64 @"),
    ("sign rule on the largest entry instead of the largest magnitude",
     "int(np.argmax(np.abs(W[k])))", "int(np.argmax(W[k]))"),
]


def _pin_calls(module):
    """Every pin of a module as (name, function, kwargs), parametrisations expanded."""
    calls = []
    for name, fn in vars(module).items():
        if not name.startswith("test_") or not callable(fn):
            continue
        marks = [m for m in getattr(fn, "pytestmark", []) if m.name == "parametrize"]
        if not marks:
            calls.append((name, fn, {}))
            continue
        assert len(marks) == 1, name
        names = [a.strip() for a in marks[0].args[0].split(",")]
        for v in marks[0].args[1]:
            calls.append((f"{name}[{v!r:.40}]", fn, dict(zip(names, v if len(names) > 1 else (v,)))))
    return calls


def _first_failing_pin(module):
    for name, fn, kw in _pin_calls(module):
        try:
            fn(**kw)
        except pytest.skip.Exception:
            continue
        except (AssertionError, ValueError):  # a failed check, or the oracle rejecting its input
            return name
    return None


def _planted(path, old, new):
    src = open(path).read()
    assert src.count(old) == 1, f"snippet to plant occurs {src.count(old)} times"
    return src.replace(old, new)


def _build_c(src, out_dir):
    os.makedirs(out_dir, exist_ok=True)
    c_path = os.path.join(out_dir, "oracle.c")
    lib_path = os.path.join(out_dir, "liboracle.so")
    open(c_path, "w").write(src)
    cmd = ["gcc", "-O1", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", c_path, "-o", lib_path, "-lm"]
    subprocess.run(cmd, check=True, capture_output=True)
    return lib_path


@pytest.fixture(scope="module")
def c_source():
    if shutil.which("gcc") is None:
        pytest.skip("gcc is needed to build the planted copies")
    return os.path.join(ORACLE_DIR, "oracle.c")


def test_pins_pass_on_the_oracle_itself():
    assert _first_failing_pin(pins) is None
    assert _first_failing_pin(pca_pins) is None


@pytest.mark.parametrize("what,old,new", C_MUTANTS, ids=[m[0] for m in C_MUTANTS])
def test_pins_catch_a_planted_c_mistake(c_source, tmp_path, monkeypatch, what, old, new):
    lib = _build_c(_planted(c_source, old, new), str(tmp_path / "mutant"))
    monkeypatch.setattr(oracle, "_lib", None)
    monkeypatch.setattr(oracle, "build", lambda force=False: lib)
    assert oracle._load()._name == lib  # the planted copy is the one the pins call
    caught_by = _first_failing_pin(pins)
    assert caught_by is not None, f"no pin fails with the planted mistake: {what}"
    print(f"{what}: caught by {caught_by}")


@pytest.mark.parametrize("what,old,new", PCA_MUTANTS, ids=[m[0] for m in PCA_MUTANTS])
def test_pins_catch_a_planted_pca_mistake(monkeypatch, what, old, new):
    src = _planted(os.path.join(ORACLE_DIR, "pca.py"), old, new)
    mutant = types.ModuleType("oracle_pca_planted")
    exec(compile(src, "oracle_pca_planted.py", "exec"), mutant.__dict__)
    monkeypatch.setattr(pca_pins, "pca", mutant)
    caught_by = _first_failing_pin(pca_pins)
    assert caught_by is not None, f"no pin fails with the planted mistake: {what}"
    print(f"{what}: caught by {caught_by}")
