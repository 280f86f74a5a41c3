"""Mistakes planted in copies of the oracle must fail at least one pin.

Each mutant is a plausible slip in the oracle's C++: for Algorithm 1 (scan
order, window bound, row or length off by one, token range, duplicate
handling, gather source, decode history alignment) and for Algorithm 3
(window bound, length range, first occurrence, threshold, sort direction, tie
order, the top-S cut, sequence boundary), and in the f-gram model oracle
(rotation direction and base, causal mask, score scale, layer-norm epsilon,
gate/up swap, a dropped residual, the output position, bf16 tie rounding,
and the absolute positions dropped, counted from the end, or added after the
first layer norm).
The copy is compiled (C++) or loaded (Python) on the CPU and the pin tests
run against it in a subprocess; they must fail.
"""

import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRCS = {"alg1": os.path.join(ROOT, "oracle", "scone_oracle.cpp"),
        "alg3": os.path.join(ROOT, "oracle", "discover_oracle.cpp")}
PINS = [os.path.join(ROOT, "tests", "test_oracle.py"),
        os.path.join(ROOT, "tests", "test_discover_oracle.py")]
MODEL_SRC = os.path.join(ROOT, "oracle", "fgram_model.py")
MODEL_PINS = os.path.join(ROOT, "tests", "test_fgram_model_oracle.py")

MODEL_MUTANTS = {
    "m_rope_direction": ("[a * c - b * s, b * c + a * s]", "[a * c + b * s, b * c - a * s]"),
    "m_rope_base": ("ROPE_BASE = 10000.0", "ROPE_BASE = 1000.0"),
    "m_no_causal_mask": ("scores = np.where(np.tril(np.ones((n, n), bool)), scores, -np.inf)",
                         "scores = scores"),
    "m_no_score_scale": ("scores = qh @ kh.T / np.sqrt(hd)", "scores = qh @ kh.T"),
    "m_ln_eps": ("LN_EPS = 1e-5", "LN_EPS = 1e-3"),
    "m_gate_up_swapped": ('mats["gate"] = gu[:, 0].reshape(f, d)', 'mats["gate"] = gu[:, 1].reshape(f, d)'),
    "m_attention_residual_dropped": ('x = r(x + o @ L["o"].T)', 'x = r(o @ L["o"].T)'),
    "m_first_position": ("f = layer_norm(x[-1:])[0]", "f = layer_norm(x[:1])[0]"),
    "m_round_half_up": ("np.round(m * 256.0)", "np.floor(m * 256.0 + 0.5)"),
    # the absolute position scheme of Appendix F
    "m_pos_dropped": ("    x0 = x0 + position_rows(W, idx.shape[0])\n", "    x0 = x0\n"),
    "m_pos_from_end": ("    return W.P[:n]\n", "    return W.P[:n][::-1]\n"),
    "m_pos_after_first_ln": [
        ("    x0 = x0 + position_rows(W, idx.shape[0])\n", "    x0 = x0\n"),
        ("        xn = r(layer_norm(x))\n        q, k, v",
         "        xn = r(layer_norm(x) + position_rows(W, x.shape[0]))\n        q, k, v")],
}

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
    # Algorithm 1
    "shortest_first": ("alg1", "for (int64_t jp = first; jp < i; ++jp) {",
                       "for (int64_t jp = i - 1; jp >= first; --jp) {"),
    "grow_until_miss": ("alg1", SCAN, GROW_UNTIL_MISS),
    "drop_longest_length": ("alg1", "int64_t first = i - (t.K - 1);", "int64_t first = i - (t.K - 2);"),
    "row_off_by_one": ("alg1", "return it->second;", "return it->second + 1;"),
    "len_off_by_one": ("alg1", "*j_out = jp;", "*j_out = jp + 1;"),
    "vocab_bound": ("alg1", "return x >= 0 && x < t.vocab;", "return x >= 0 && x <= t.vocab;"),
    "duplicates_accepted": ("alg1", "      delete t;\n      return -3;", "      (void)0;"),
    "fallback_wrong_token": ("alg1", "T + (int64_t)seq[i] * d", "T + (int64_t)seq[i > 0 ? i - 1 : 0] * d"),
    "fgram_row_shift": ("alg1", "F + r * d", "F + (r > 0 ? r - 1 : r) * d"),
    "decode_history_left_aligned": ("alg1", "hist + s * hist_stride + (hist_stride - h)",
                                    "hist + s * hist_stride"),
    # Algorithm 3
    "d_last_window_dropped": ("alg3", "for (int64_t p = 0; p + n <= L; ++p)",
                              "for (int64_t p = 0; p + n < L; ++p)"),
    "d_longest_length_dropped": ("alg3", "for (int32_t n = 2; n <= K; ++n)",
                                 "for (int32_t n = 2; n < K; ++n)"),
    "d_last_occurrence": ("alg3", "if (e.count == 0) e.first = b * L + p;",
                          "e.first = b * L + p;"),
    "d_threshold_strict": ("alg3", "if (kv.second.count < min_count) continue;",
                           "if (kv.second.count <= min_count) continue;"),
    "d_least_frequent_first": ("alg3", "if (a.count != b.count) return a.count > b.count;",
                               "if (a.count != b.count) return a.count < b.count;"),
    "d_ties_longest_first": ("alg3", "if (a.gram.size() != b.gram.size()) return a.gram.size() < "
                             "b.gram.size();\n    return a.first < b.first;\n  });\n  if",
                             "if (a.gram.size() != b.gram.size()) return a.gram.size() > "
                             "b.gram.size();\n    return a.first < b.first;\n  });\n  if"),
    "d_cut_one_short": ("alg3", "all.resize((size_t)S);", "all.resize((size_t)(S > 0 ? S - 1 : 0));"),
    "d_cross_sequences": ("alg3", "for (int64_t p = 0; p + n <= L; ++p) {\n        Entry& e = "
                          "counts[std::vector<int32_t>(seq + p, seq + p + n)];",
                          "for (int64_t p = 0; p + n <= L + (b + 1 < B ? n - 1 : 0); ++p) {\n"
                          "        Entry& e = counts[std::vector<int32_t>(seq + p, seq + p + n)];"),
    "d_vocab_bound": ("alg3", "if (tok[i] < 0 || tok[i] >= vocab) return -2;",
                      "if (tok[i] < 0 || tok[i] > vocab) return -2;"),
}


def _run_pins(lib):
    env = dict(os.environ, SCONE_ORACLE_LIB=lib)
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        *PINS], cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode, r.stdout[-2000:]


def _compile(tmp_path, which=None, old=None, new=None):
    cpps = []
    for key, path in sorted(SRCS.items()):
        src = open(path).read()
        if key == which:
            assert old in src, f"mutation site not found: {old[:60]}"
            src = src.replace(old, new)
        cpp = tmp_path / f"{key}.cpp"
        cpp.write_text(src)
        cpps.append(str(cpp))
    lib = str(tmp_path / "liboracle_copy.so")
    subprocess.run(["g++", "-O1", "-std=c++17", "-fPIC", "-shared", *cpps, "-o", lib], check=True)
    return lib


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    which, old, new = MUTANTS[name]
    rc, log = _run_pins(_compile(tmp_path, which, old, new))
    assert rc != 0, f"mutant {name} passed every pin:\n{log}"


def test_unmutated_copy_passes(tmp_path):
    rc, log = _run_pins(_compile(tmp_path))
    assert rc == 0, log


@pytest.mark.parametrize("name", sorted(MODEL_MUTANTS))
def test_model_mutant_is_caught(name, tmp_path):
    edits = MODEL_MUTANTS[name]
    src = open(MODEL_SRC).read()
    for old, new in ([edits] if isinstance(edits, tuple) else edits):
        assert src.count(old) == 1, f"mutation site for {name} not found once"
        src = src.replace(old, new)
    path = tmp_path / "fgram_model_mut.py"
    path.write_text(src)
    env = dict(os.environ, SCONE_FGRAM_ORACLE_FILE=str(path))
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        MODEL_PINS], cwd=ROOT, env=env, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode != 0, f"mutant {name} passed every pin:\n{r.stdout[-2000:]}"
