"""The seeded input generator: determinism, shapes and structure."""
import numpy as np
import pytest

from paper_2607_18839_gb300 import workloads as W


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.0 + 2**-8, 1.0 + 3 * 2**-8, -2.5, 0.0, 3.0e38], dtype=np.float32)
    b = W.f32_to_bf16_bits(x)
    back = W.bf16_bits_to_f32(b)
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: even mantissa -> 1.0
    assert back[0] == 1.0 and back[1] == 1.0 and back[2] == 1.0 + 2**-6
    assert back[3] == -2.5 and back[4] == 0.0


@pytest.mark.parametrize("name", ["c1", "c2", "c3"])
def test_configs_are_deterministic_and_well_formed(name):
    a = W.make_config(name)
    b = W.make_config(name)
    assert np.array_equal(a.q, b.q) and np.array_equal(a.page_table, b.page_table)
    assert a.q.shape == (a.B * a.m, a.H_q, a.D)
    assert a.prefix_k.shape == (a.prefix_tokens, a.H_kv, a.D)
    assert a.k_cache.shape == (a.num_pages, W.PAGE, a.H_kv, a.D)
    assert np.all((a.page_table >= 0) & (a.page_table < a.num_pages))
    used = []
    for bb in range(a.B):
        n = (int(a.branch_len[bb]) + W.PAGE - 1) // W.PAGE
        used.extend(a.page_table[bb, :n].tolist())
    assert len(used) == len(set(used))  # no physical page shared between branches


def test_config_shapes_match_the_presets():
    c4 = W.make_config("c4")
    assert c4.n_docs == 32 and c4.B == 32 * 24 and c4.m == 8 and (c4.H_q, c4.H_kv) == (16, 2)
    P = np.diff(c4.prefix_cu)
    assert P.min() >= 1024 and P.max() <= 3072
    c5 = W.make_config("c5")
    s = c5.branch_len - c5.m
    assert s.min() >= 8 and s.max() <= 2048 and c5.B == 256


def test_mix_drafts_rate():
    t = np.arange(40000, dtype=np.int32).reshape(10000, 4) % 32000
    d = W.mix_drafts(t, 32000, 0.7, seed=3)
    rate = np.mean(d == t)
    assert 0.68 < rate < 0.72
