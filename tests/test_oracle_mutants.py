"""Mistakes planted in copies of the oracle must fail at least one pin.

Each mutant is a plausible slip in the oracle's C++ (scan order, window
bound, row or length off by one, token range, duplicate handling, gather
source, decode history alignment). The copy is compiled on the CPU and the
pin tests in test_oracle.py run against it in a subprocess; they must fail.
"""

import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "scone_oracle.cpp")

SCAN = """  for (int64_t jp = first; jp < i; ++jp) {
    const std::vector<int32_t> window(seq + jp, seq + i + 1);
    if (queries) ++*queries;
    const auto it = t.fgram_row.find(window);
    if (it != t.fgram_row.end()) {
      *j_out = jp;
      return it->second;
    }
  }
  *j_out = i;
  return -1;"""

GROW_UNTIL_MISS = """  int64_t best = -1;
  *j_out = i;
  for (int64_t jp = i - 1; jp >= first; --jp) {
    const std::vector<int32_t> window(seq + jp, seq + i + 1);
    if (queries) ++*queries;
    const auto it = t.fgram_row.find(window);
    if (it == t.fgram_row.end()) break;
    best = it->second;
    *j_out = jp;
  }
  return best;"""

MUTANTS = {
    "shortest_first": ("for (int64_t jp = first; jp < i; ++jp) {",
                       "for (int64_t jp = i - 1; jp >= first; --jp) {"),
    "grow_until_miss": (SCAN, GROW_UNTIL_MISS),
    "drop_longest_length": ("int64_t first = i - (t.K - 1);", "int64_t first = i - (t.K - 2);"),
    "row_off_by_one": ("return it->second;", "return it->second + 1;"),
    "len_off_by_one": ("*j_out = jp;", "*j_out = jp + 1;"),
    "vocab_bound": ("return x >= 0 && x < t.vocab;", "return x >= 0 && x <= t.vocab;"),
    "duplicates_accepted": ("      delete t;\n      return -3;", "      (void)0;"),
    "fallback_wrong_token": ("T + (int64_t)seq[i] * d", "T + (int64_t)seq[i > 0 ? i - 1 : 0] * d"),
    "fgram_row_shift": ("F + r * d", "F + (r > 0 ? r - 1 : r) * d"),
    "decode_history_left_aligned": ("hist + s * hist_stride + (hist_stride - h)",
                                    "hist + s * hist_stride"),
}


def _run_pins(lib):
    env = dict(os.environ, SCONE_ORACLE_LIB=lib)
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode, r.stdout[-2000:]


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert old in src, f"mutation site for {name} not found"
    mutated = src.replace(old, new)
    cpp = tmp_path / "mut.cpp"
    cpp.write_text(mutated)
    lib = str(tmp_path / "libmut.so")
    subprocess.run(["g++", "-O1", "-std=c++17", "-fPIC", "-shared", str(cpp), "-o", lib],
                   check=True)
    rc, log = _run_pins(lib)
    assert rc != 0, f"mutant {name} passed every pin:\n{log}"


def test_unmutated_copy_passes(tmp_path):
    cpp = tmp_path / "same.cpp"
    cpp.write_text(open(SRC).read())
    lib = str(tmp_path / "libsame.so")
    subprocess.run(["g++", "-O1", "-std=c++17", "-fPIC", "-shared", str(cpp), "-o", lib],
                   check=True)
    rc, log = _run_pins(lib)
    assert rc == 0, log
