"""The pins are sharp: each plausible mistake planted in a copy of the oracle
(compiled on the CPU into a temporary library) fails at least one pin.

The mutated copies live only in pytest's tmp_path; the committed oracle is
untouched.  Every mutation keeps all memory accesses in bounds.
"""
import ctypes
import os
import subprocess

import pytest

import oracle
import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "hpd_oracle.c")

# (name, original text, mutated text, replace every occurrence)
MUTATIONS = [
    ("causal rule off by one", "const int last_private = L_b - m + i;",
     "const int last_private = L_b - m + i - 1;", False),
    ("causal rule lets the whole step see itself", "const int last_private = L_b - m + i;",
     "const int last_private = L_b - 1;", False),
    ("kv head interleaved instead of grouped", "const int g = h / G;",
     "const int g = h % H_kv;", False),
    ("scale dropped", "s[n++] = scale * dot;", "s[n++] = dot;", True),
    ("lse in base 2", "M + log(denom)", "M + log2(denom)", False),
    ("fork-position prefix ignored", "int P_b = branch_prefix_len ? branch_prefix_len[b] : P_d;",
     "int P_b = P_d;", False),
    ("page slot transposed", "(((long)page * ORACLE_PAGE + j % ORACLE_PAGE) * H_kv + g) * D",
     "(((long)page * ORACLE_PAGE + (j / ORACLE_PAGE) % ORACLE_PAGE) * H_kv + g) * D", True),
    ("prefix term dropped from the weights", "for (int j = 0; j < P_b; ++j, ++t) {",
     "for (int j = 0; j < 0; ++j, ++t) {", False),
    ("max not subtracted in the weights", "const double w = exp(s[t] - M) / denom;",
     "const double w = exp(s[t]) / denom;", True),
    ("paged prefix slot transposed",
     "ORACLE_PAGE + (j) % ORACLE_PAGE ", "ORACLE_PAGE + ((j) / ORACLE_PAGE) % ORACLE_PAGE ", False),
    ("paged prefix reads page 0's table row",
     "prefix_page_table[(long)d * max_prefix_pages + (j) / ORACLE_PAGE]",
     "prefix_page_table[(long)0 * max_prefix_pages + (j) / ORACLE_PAGE]", False),
    ("argmax keeps the last of equal maxima", "if (!seen || x > best_val) {",
     "if (!seen || x >= best_val) {", False),
    ("accepted length counts the bonus token", "accepted_len[b] = k;",
     "accepted_len[b] = k < m ? k + 1 : k;", False),
]

PIN_TESTS = [
    lambda: [pins.test_oracle_matches_explicit_mask_brute_force(c) for c in range(6)],
    pins.test_zero_query_gives_mean_of_visible_values_and_log_count,
    pins.test_constant_values_give_that_value,
    pins.test_empty_suffix_single_query_is_plain_prefix_attention,
    pins.test_two_keys_closed_form_scale_and_natural_log,
    pins.test_gqa_groups_contiguous_query_heads,
    pins.test_no_visible_key_gives_zero_and_minus_inf,
    pins.test_causality_among_the_m_queries,
    lambda: [pins.test_paged_prefix_matches_brute_force_on_the_same_keys(c) for c in range(6)],
    pins.test_paged_prefix_follows_the_table,
    pins.test_accept_closed_forms,
    pins.test_accept_ties_lowest_index_and_nan_ignored,
    pins.test_accept_matches_numpy_argmax_brute_force,
]


def _compile(tmp_path, text, tag):
    src = tmp_path / f"mut_{tag}.c"
    lib = tmp_path / f"libmut_{tag}.so"
    src.write_text(text)
    subprocess.run(["gcc", "-O1", "-fopenmp", "-fPIC", "-shared", "-std=c11", "-o", str(lib),
                    str(src), "-lm"], check=True)
    return str(lib)


def _bind(path):
    lib = ctypes.CDLL(path)
    P, I = ctypes.c_void_p, ctypes.c_int
    lib.oracle_branch_attn.restype = I
    lib.oracle_branch_attn.argtypes = [P] * 10 + [I] * 8 + [ctypes.c_double, P, I, I, P, P, P, I]
    lib.oracle_pmtp_accept.restype = None
    lib.oracle_pmtp_accept.argtypes = [P, P, I, I, I, P, P]
    lib.oracle_max_threads.restype = I
    return lib


@pytest.mark.parametrize("k", range(len(MUTATIONS)), ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_fails_a_pin(k, tmp_path, monkeypatch):
    name, old, new, every = MUTATIONS[k]
    text = open(SRC).read()
    assert old in text, f"mutation anchor for {name!r} not found"
    text = text.replace(old, new) if every else text.replace(old, new, 1)
    lib = _bind(_compile(tmp_path, text, k))
    monkeypatch.setattr(oracle, "_lib", lib)
    failed = 0
    for t in PIN_TESTS:
        try:
            t()
        except (AssertionError, ValueError):
            failed += 1
    assert failed >= 1, f"no pin caught: {name}"
