"""Pins for the float64 attention oracle: closed forms, invariants and a
pure-Python brute force on tiny inputs (none of them re-runs the oracle's
own formula)."""
import itertools
import math
import random

import numpy as np
import pytest

from oracle import attention as A
from conftest import read_golden


def _rand(rng, *shape, scale=1.0):
    return rng.standard_normal(shape) * scale


def test_two_keys_closed_form():
    g = {k: float(v) for k, v in read_golden("two_key_softmax.txt")}
    q = np.array([[2.0, 0, 0, 0]])
    k = np.array([[[1.0, 0, 0, 0]], [[0.0, 0, 0, 0]]])
    v = np.array([[[1.0, 0, 0, 0]], [[0.0, 1, 0, 0]]])
    o, lse = A.decode(q, k, v)
    assert o[0, 0] == pytest.approx(g["o0"], abs=1e-15)
    assert o[0, 1] == pytest.approx(g["o1"], abs=1e-15)
    assert o[0, 2] == 0 and o[0, 3] == 0
    assert lse[0] == pytest.approx(g["lse"], abs=1e-15)


def test_single_key_returns_its_value():
    rng = np.random.default_rng(1)
    q = _rand(rng, 4, 8)
    k = _rand(rng, 1, 2, 8)
    v = _rand(rng, 1, 2, 8)
    o, lse = A.decode(q, k, v)
    for h in range(4):
        g = h // 2
        np.testing.assert_array_equal(o[h], v[0, g])
        # lse of one key is its score: q.k/sqrt(D)
        s = sum(q[h, d] * k[0, g, d] for d in range(8)) / math.sqrt(8)
        assert lse[h] == pytest.approx(s, abs=1e-13)


def test_identical_keys_give_mean_value():
    rng = np.random.default_rng(2)
    n, D = 7, 16
    q = _rand(rng, 2, D)
    key = _rand(rng, D)
    k = np.tile(key, (n, 1, 1))
    v = _rand(rng, n, 1, D)
    o, lse = A.decode(q, k, v)
    for h in range(2):
        np.testing.assert_allclose(o[h], v[:, 0].mean(axis=0), atol=1e-14)
        s = float(q[h] @ key) / math.sqrt(D)
        assert lse[h] == pytest.approx(s + math.log(n), abs=1e-13)


def test_zero_query_is_uniform():
    rng = np.random.default_rng(3)
    n, D = 11, 8
    k = _rand(rng, n, 1, D)
    v = _rand(rng, n, 1, D)
    o, lse = A.decode(np.zeros((1, D)), k, v)
    np.testing.assert_allclose(o[0], v[:, 0].mean(axis=0), atol=1e-14)
    assert lse[0] == pytest.approx(math.log(n), abs=1e-14)


def test_gqa_heads_read_contiguous_kv_groups():
    # Hq = 6, Hkv = 3 -> G = 2: heads {0,1} -> kv 0, {2,3} -> kv 1, {4,5} -> kv 2.
    # Each kv head holds identical keys and a constant value equal to its index,
    # so head h must return floor(h / 2) everywhere.
    D, n = 4, 5
    rng = np.random.default_rng(4)
    q = _rand(rng, 6, D)
    k = np.zeros((n, 3, D))
    v = np.zeros((n, 3, D))
    for g in range(3):
        k[:, g, :] = _rand(rng, D)
        v[:, g, :] = float(g)
    o, _ = A.decode(q, k, v)
    for h in range(6):
        np.testing.assert_allclose(o[h], np.full(D, float(h // 2)), atol=1e-14)


def _brute(q, k, v):
    """Softmax attention with scalar Python arithmetic (math.exp, math.fsum)."""
    Hq, D = len(q), len(q[0])
    n, Hkv = len(k), len(k[0])
    G = Hq // Hkv
    out, lses = [], []
    for h in range(Hq):
        g = h // G
        scores = [math.fsum(q[h][d] * k[j][g][d] for d in range(D)) / math.sqrt(D) for j in range(n)]
        mx = max(scores)
        z = math.fsum(math.exp(s - mx) for s in scores)
        lse = mx + math.log(z)
        out.append([math.fsum(math.exp(scores[j] - lse) * v[j][g][d] for j in range(n)) for d in range(D)])
        lses.append(lse)
    return out, lses


@pytest.mark.parametrize("n,Hq,Hkv,D", [(1, 2, 1, 2), (3, 4, 2, 4), (6, 4, 1, 8), (5, 6, 3, 2)])
def test_brute_force_tiny(n, Hq, Hkv, D):
    r = random.Random(n * 1000 + Hq * 100 + Hkv * 10 + D)
    q = [[r.gauss(0, 1.5) for _ in range(D)] for _ in range(Hq)]
    k = [[[r.gauss(0, 1.5) for _ in range(D)] for _ in range(Hkv)] for _ in range(n)]
    v = [[[r.gauss(0, 1) for _ in range(D)] for _ in range(Hkv)] for _ in range(n)]
    o_ref, lse_ref = _brute(q, k, v)
    o, lse = A.decode(np.array(q), np.array(k), np.array(v))
    np.testing.assert_allclose(o, np.array(o_ref), rtol=0, atol=1e-13)
    np.testing.assert_allclose(lse, np.array(lse_ref), rtol=0, atol=1e-13)


def test_key_order_does_not_matter():
    rng = np.random.default_rng(5)
    q, k, v = _rand(rng, 4, 16), _rand(rng, 30, 2, 16), _rand(rng, 30, 2, 16)
    perm = rng.permutation(30)
    o1, l1 = A.decode(q, k, v)
    o2, l2 = A.decode(q, k[perm], v[perm])
    np.testing.assert_allclose(o1, o2, atol=1e-13)
    np.testing.assert_allclose(l1, l2, atol=1e-13)


def test_value_linearity():
    rng = np.random.default_rng(6)
    q, k, v = _rand(rng, 4, 16), _rand(rng, 9, 2, 16), _rand(rng, 9, 2, 16)
    o1, l1 = A.decode(q, k, v)
    o2, l2 = A.decode(q, k, 3.0 * v - 1.0)
    np.testing.assert_allclose(o2, 3.0 * o1 - 1.0, atol=1e-13)
    np.testing.assert_array_equal(l1, l2)


@pytest.mark.parametrize("cuts", [(1,), (5, 6), (1, 2, 3, 30), (17,)])
def test_lse_split_equals_unsplit(cuts):
    rng = np.random.default_rng(7)
    n = 31
    q, k, v = _rand(rng, 8, 16, scale=2), _rand(rng, n, 2, 16), _rand(rng, n, 2, 16)
    edges = [0, *cuts, n]
    parts = [A.decode(q, k[a:b], v[a:b]) for a, b in zip(edges, edges[1:])]
    o, lse = A.combine(parts)
    o_ref, lse_ref = A.decode(q, k, v)
    np.testing.assert_allclose(o, o_ref, atol=1e-12)
    np.testing.assert_allclose(lse, lse_ref, atol=1e-12)


def test_combine_ignores_empty_partials():
    rng = np.random.default_rng(8)
    q, k, v = _rand(rng, 2, 4), _rand(rng, 5, 1, 4), _rand(rng, 5, 1, 4)
    o, lse = A.decode(q, k, v)
    empty = (np.full_like(o, 123.0), np.full_like(lse, -np.inf))
    o2, lse2 = A.combine([(o, lse), empty])
    np.testing.assert_allclose(o2, o, atol=1e-15)
    np.testing.assert_allclose(lse2, lse, atol=1e-15)


def test_empty_suffix_branch_equals_main():
    # A branch whose suffix is empty sees exactly main's context.
    rng = np.random.default_rng(9)
    k, v, q = _rand(rng, 40, 2, 8), _rand(rng, 40, 2, 8), _rand(rng, 4, 8)
    suffix_k, suffix_v = k[:0], v[:0]
    o_main, l_main = A.decode(q, k, v)
    o_b, l_b = A.decode(q, np.concatenate([k, suffix_k]), np.concatenate([v, suffix_v]))
    np.testing.assert_array_equal(o_main, o_b)
    np.testing.assert_array_equal(l_main, l_b)


def test_decode_rejects_empty_context():
    with pytest.raises(ValueError):
        A.decode(np.zeros((1, 4)), np.zeros((0, 1, 4)), np.zeros((0, 1, 4)))


# ---- merge prefill -------------------------------------------------------

def test_merge_single_row_equals_decode_after_append():
    rng = np.random.default_rng(10)
    L0 = 23
    k, v = _rand(rng, L0 + 1, 2, 8), _rand(rng, L0 + 1, 2, 8)
    q = _rand(rng, 1, 4, 8)
    o, lse = A.merge_prefill(q, k, v, L0)
    o2, l2 = A.decode(q[0], k, v)
    np.testing.assert_array_equal(o[0], o2)
    np.testing.assert_array_equal(lse[0], l2)


def test_merge_is_causal_and_last_row_sees_everything():
    rng = np.random.default_rng(11)
    L0, T = 20, 9
    k, v = _rand(rng, L0 + T, 2, 8), _rand(rng, L0 + T, 2, 8)
    q = _rand(rng, T, 4, 8)
    o, lse = A.merge_prefill(q, k, v, L0)
    # perturbing rows after L0 + i leaves row i unchanged
    k2, v2 = k.copy(), v.copy()
    k2[L0 + 4:] += 5.0
    v2[L0 + 4:] -= 7.0
    o2, l2 = A.merge_prefill(q, k2, v2, L0)
    np.testing.assert_array_equal(o[:4], o2[:4])
    assert not np.allclose(o[5:], o2[5:])
    # last row equals a decode over the whole context
    o3, l3 = A.decode(q[-1], k, v)
    np.testing.assert_array_equal(o[-1], o3)
    # row i with a hand-built causal context
    i = 6
    o4, _ = A.decode(q[i], k[: L0 + i + 1], v[: L0 + i + 1])
    np.testing.assert_array_equal(o[i], o4)


def test_merge_row_subset_matches_full():
    rng = np.random.default_rng(12)
    L0, T = 5, 12
    k, v = _rand(rng, L0 + T, 1, 4), _rand(rng, L0 + T, 1, 4)
    q = _rand(rng, T, 2, 4)
    o, lse = A.merge_prefill(q, k, v, L0)
    rows = [0, 7, 11]
    os_, ls_ = A.merge_prefill(q, k, v, L0, rows=rows)
    np.testing.assert_array_equal(o[rows], os_)
    np.testing.assert_array_equal(lse[rows], ls_)
