"""Pins for the fp64 oracle: each test checks it against something other than itself.

Sources of truth used here:
  * values derived by hand from Eq. (pbb) and Eq. (attention) at the size of
    Fig. 1 (tests/golden/hand_b4.json);
  * numbers printed in the paper: score counts at n = 8192 (Sec. 3 and the
    table of Appendix A.5), the support count of Eq. (pbb_cache_support), its
    phase mean, and the ring size (Appendix F.1) (tests/golden/paper_counts.json);
  * a second definition of the support from the paper, the interval form
    [a(t), t] of Eq. (pbb_relay), and the proof of the ring proposition;
  * special cases with a closed form (t = 0, q = 0) and library routines
    (scipy softmax) on tiny inputs; the fusion identity of Eq. (lse).
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def interval_start(t, b):
    """a(t) = max(0, h(floor(t/h) - 1)), the interval form of Eq. (pbb_relay)."""
    h = b // 2
    return max(0, h * (t // h - 1))


# ---------------------------------------------------------------- support --


def test_hand_supports(oracle_mod):
    g = load("hand_b4.json")
    b = g["b"]
    for t_str, sup in g["supports"].items():
        t = int(t_str)
        got = [s for s in range(t + 1) if oracle_mod.in_support(t, s, b)]
        assert got == sup, t


@pytest.mark.parametrize("b", [2, 4, 6, 8, 10, 16, 32, 64])
def test_support_matches_interval_form(oracle_mod, b):
    for t in range(8 * b):
        a = interval_start(t, b)
        for s in range(-2, t + 3):
            assert oracle_mod.in_support(t, s, b) == (a <= s <= t), (b, t, s)


def test_support_interval_form_large_block(oracle_mod):
    b = 128
    rng = np.random.default_rng(5)
    for t in list(range(0, 3 * b)) + list(rng.integers(0, 1 << 20, 64)):
        t = int(t)
        a = interval_start(t, b)
        for s in range(max(-1, a - 70), t + 2):
            assert oracle_mod.in_support(t, s, b) == (a <= s <= t)


@pytest.mark.parametrize("b", [2, 4, 8, 12, 64, 128, 1024])
def test_support_count_closed_form(oracle_mod, b):
    """Eq. (pbb_cache_support): |A(t)| = h + 1 + (t mod h) after the first block."""
    h = b // 2
    ts = list(range(min(8 * b, 3000)))
    for t in ts:
        n = oracle_mod.support_count(t, b)
        if t >= b:
            assert n == h + 1 + (t % h), (b, t)
            assert n <= b
        else:
            assert n == t + 1, (b, t)  # first block: no bridge (p = 0)


def test_phase_mean_support(oracle_mod):
    """Appendix F.1: the steady-state phase average is (3h+1)/2 = 96.5 at h = 64."""
    g = load("paper_counts.json")
    b = g["b"]
    mean = np.mean([oracle_mod.support_count(t, b) for t in range(5 * b, 6 * b)])
    assert mean == g["phase_mean_support_h64"]


def test_score_counts_at_8192(oracle_mod):
    """Exact score counts of Sec. 3 / Appendix A.5 at n = 8192, b = 128, h = 64."""
    g = load("paper_counts.json")
    n, b = g["n"], g["b"]
    e_pbb = sum(oracle_mod.support_count(t, b) for t in range(n))
    assert e_pbb == g["E_PBB"]
    # every within-block causal score is kept: sum_t (r+1) is the Block-128 count,
    # and the remainder is the cross-block (bridge) count the paper prints.
    e_block = sum(t % b + 1 for t in range(n))
    assert e_block == g["E_Block"]
    assert e_pbb - e_block == g["cross_block_PBB"]
    # the SWA-128 window counts of the same table
    e_swa = sum(min(t + 1, b) for t in range(n))
    assert e_swa == g["E_SWA"] and e_swa - e_block == g["cross_block_SWA"]
    # 20-layer 3:1 hybrid: 15 PBB layers and 5 Full layers
    e_full = n * (n + 1) // 2
    assert e_full == g["E_Full"]
    assert 15 * e_pbb + 5 * e_full == g["hybrid_20_layer_PBB"]
    assert 20 * e_full == g["hybrid_20_layer_Full"]
    assert round(100 * g["hybrid_20_layer_PBB"] / g["hybrid_20_layer_Full"], 2) == g[
        "hybrid_fraction_percent"]


def test_pbb_subset_of_swa(oracle_mod):
    """Sec. 3 / App. A.4: every PBB edge has distance t - s < w = 2h = b."""
    b = 16
    for t in range(10 * b):
        for s in range(t + 1):
            if oracle_mod.in_support(t, s, b):
                assert t - s < b


@pytest.mark.parametrize("n,b", [(1024, 128), (4096, 1024), (8192, 128), (2048, 64)])
def test_score_budget_closed_form(oracle_mod, n, b):
    """Appendix A.5: E_PBB = n(b+1)/2 + (n/b - 1) h^2 for n divisible by b."""
    h = b // 2
    assert sum(oracle_mod.support_count(t, b) for t in range(n)) == n * (b + 1) // 2 + (n // b - 1) * h * h


# -------------------------------------------------------------- attention --


def _frac(x):
    return float(Fraction(x))


def test_hand_attention_values(oracle_mod):
    g = load("hand_b4.json")
    b, T = g["b"], 12
    s = np.arange(T, dtype=np.float64)
    v = s.reshape(1, 1, T, 1)
    cases = {
        "uniform weights": (0.0, np.zeros_like(s)),
        "weights 3 and 1": (1.0, np.where(s % 2 == 0, math.log(3.0), 0.0)),
    }
    for case in g["cases"]:
        qv, kv = cases[case["name"]]
        k = kv.reshape(1, 1, T, 1)
        for t in range(T):
            q = np.full((1, 1, 1), qv)
            o = oracle_mod.attend(q, k, v, s0=[0], t=[t], b=b)
            assert abs(o[0, 0, 0] - _frac(case["out"][t])) < 1e-12, (case["name"], t)


def _rand_problem(rng, batch, Hq, Hkv, d, n_hist):
    q = rng.standard_normal((batch, Hq, d))
    k = rng.standard_normal((batch, Hkv, n_hist, d))
    v = rng.standard_normal((batch, Hkv, n_hist, d))
    return q, k, v


def test_first_token_returns_its_value(oracle_mod):
    """t = 0: the support is {0}, so o = v_0 exactly whatever q and k are."""
    rng = np.random.default_rng(0)
    q, k, v = _rand_problem(rng, 3, 8, 2, 16, 1)
    o = oracle_mod.attend(q, k, v, s0=0, t=0, b=8)
    for j in range(8):
        assert np.array_equal(o[:, j], v[:, j // 4, 0])


def test_zero_query_gives_support_mean(oracle_mod):
    """q = 0: equal weights, o is the mean of V over [a(t), t]."""
    rng = np.random.default_rng(1)
    b, d, n = 8, 5, 50
    _, k, v = _rand_problem(rng, 1, 2, 1, d, n)
    q = np.zeros((1, 2, d))
    for t in range(n):
        o = oracle_mod.attend(q, k, v, s0=0, t=t, b=b)
        ref = v[0, 0, interval_start(t, b):t + 1].mean(axis=0)
        assert np.allclose(o[0, 0], ref, rtol=0, atol=1e-13)


def test_matches_scipy_softmax(oracle_mod):
    """Tiny random problems: softmax (scipy) over the interval-form support."""
    from scipy.special import softmax

    rng = np.random.default_rng(2)
    batch, Hq, Hkv, d, b, n = 2, 6, 2, 4, 8, 41
    q, k, v = _rand_problem(rng, batch, Hq, Hkv, d, n)
    ts = np.array([17, 40])
    o = oracle_mod.attend(q, k, v, s0=0, t=ts, b=b)
    for bi in range(batch):
        t = int(ts[bi])
        a = interval_start(t, b)
        for j in range(Hq):
            kv = j // (Hq // Hkv)
            z = k[bi, kv, a:t + 1] @ q[bi, j] / math.sqrt(d)
            ref = softmax(z) @ v[bi, kv, a:t + 1]
            assert np.allclose(o[bi, j], ref, rtol=1e-13, atol=1e-13)


def test_lse_fusion_of_block_and_bridge(oracle_mod):
    """Eq. (lse): attention on the block part and on the bridge part, fused, is the union."""
    rng = np.random.default_rng(3)
    b, d, n = 16, 8, 80
    h = b // 2
    q, k, v = _rand_problem(rng, 1, 1, 1, d, n)
    for t in range(b, n):
        p = b * (t // b)
        r = t - p
        parts = [np.arange(p, t + 1)]
        if r < h:
            parts.append(np.arange(p - h, p))
        logz, outs = [], []
        for idx in parts:
            z = k[0, 0, idx] @ q[0, 0] / math.sqrt(d)
            m = z.max()
            w = np.exp(z - m)
            logz.append(m + math.log(w.sum()))
            outs.append(w @ v[0, 0, idx] / w.sum())
        if len(parts) == 1:
            ref = outs[0]
        else:
            m = max(logz)
            e1, e2 = math.exp(logz[0] - m), math.exp(logz[1] - m)
            ref = (e1 * outs[0] + e2 * outs[1]) / (e1 + e2)
        o = oracle_mod.attend(q, k, v, s0=0, t=t, b=b)
        assert np.allclose(o[0, 0], ref, rtol=1e-12, atol=1e-12), t


def test_gqa_contiguous_grouping(oracle_mod):
    """Query head j reads KV head j // (Hq/Hkv)."""
    Hq, Hkv, d, n = 8, 4, 3, 5
    k = np.zeros((1, Hkv, n, d))
    v = np.zeros((1, Hkv, n, d))
    for kv in range(Hkv):
        v[0, kv] = kv + 1.0
    q = np.random.default_rng(4).standard_normal((1, Hq, d))
    o = oracle_mod.attend(q, k, v, s0=0, t=n - 1, b=4)
    for j in range(Hq):
        assert np.all(o[0, j] == j // 2 + 1.0)


def test_window_must_cover_support(oracle_mod):
    """The oracle refuses, rather than guess, when a needed source is not in the window."""
    rng = np.random.default_rng(6)
    b, d = 8, 4
    q, k, v = _rand_problem(rng, 1, 1, 1, d, 4)
    t = 9  # p = 8, r = 1 < h: support is [4, 9], 6 positions
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.attend(q, k, v, s0=6, t=t, b=b)
    k2 = rng.standard_normal((1, 1, 6, d))
    v2 = rng.standard_normal((1, 1, 6, d))
    oracle_mod.attend(q, k2, v2, s0=4, t=t, b=b)


def test_empty_bridge_equals_block_attention(oracle_mod):
    """r >= h (or p = 0): no bridge, the output is plain block-prefix attention."""
    from scipy.special import softmax

    rng = np.random.default_rng(7)
    b, d, n = 8, 4, 40
    q, k, v = _rand_problem(rng, 1, 1, 1, d, n)
    for t in range(n):
        p, r = b * (t // b), t % b
        if p > 0 and r < b // 2:
            continue
        z = k[0, 0, p:t + 1] @ q[0, 0] / math.sqrt(d)
        ref = softmax(z) @ v[0, 0, p:t + 1]
        o = oracle_mod.attend(q, k, v, s0=0, t=t, b=b)
        assert np.allclose(o[0, 0], ref, rtol=1e-13, atol=1e-13)


# ------------------------------------------------------------------- ring --


def test_hand_ring_slots(oracle_mod):
    g = load("hand_b4.json")
    b = g["b"]
    ring = oracle_mod.RingSim(1, 1, 1, b, 4)
    one = np.zeros((1, 1, 1), dtype=np.float32)
    for t in range(7):
        ring.append(one, one, t)
        if str(t) in g["ring"]["after_t"]:
            assert ring.tags[0].tolist() == g["ring"]["after_t"][str(t)]


@pytest.mark.parametrize("b", list(range(2, 66, 2)) + [128, 256])
def test_ring_holds_exactly_the_support(oracle_mod, b):
    """Appendix F.1 proposition, exhaustively: after appending t, every source of
    A(t) sits in its own slot, and the position overwritten (t - b) is older than a(t)."""
    ring = oracle_mod.RingSim(1, 1, 1, b, 2)
    z = np.zeros((1, 1, 1), dtype=np.uint16)
    for t in range(8 * b):
        ring.append(z, z, t)
        a = interval_start(t, b)
        support = [s for s in range(t + 1) if oracle_mod.in_support(t, s, b)]
        assert support == list(range(a, t + 1))
        assert len(support) <= b
        slots = [s % b for s in support]
        assert len(set(slots)) == len(slots)
        for s in support:
            assert ring.tags[0, s % b] == s
        if t >= b:
            assert t - b < a


def test_ring_bytes_and_untouched_slots(oracle_mod):
    """Slots never written stay zero; written slots hold the exact element bits."""
    import torch

    b, d = 8, 4
    ring = oracle_mod.RingSim(2, 3, d, b, 2)
    g = torch.Generator().manual_seed(0)
    for t in range(5):
        k = torch.randn(2, 3, d, generator=g).bfloat16()
        v = torch.randn(2, 3, d, generator=g).bfloat16()
        ring.append(k, v, [t, t + 1])
    kb = ring.k.view(np.uint16)
    assert np.all(kb[0, :, 5:] == 0) and np.all(kb[1, :, 6:] == 0)
    assert np.array_equal(kb[1, :, 5], k[1].view(torch.int16).numpy().view(np.uint16))


@pytest.mark.parametrize("elem", [2, 4])
def test_ring_indexed_equals_full_history(oracle_mod, elem):
    """Appendix F.1: attention read from the b-slot ring over [a(t), t] equals the
    brute-force evaluation over the whole uncompressed history."""
    import torch

    g = torch.Generator().manual_seed(11)
    batch, Hq, Hkv, d, b, T = 3, 8, 2, 16, 16, 70
    dt = torch.bfloat16 if elem == 2 else torch.float32
    K = torch.randn(batch, Hkv, T, d, generator=g).to(dt)
    V = torch.randn(batch, Hkv, T, d, generator=g).to(dt)
    offs = [0, 3, 9]  # ragged: sequence bi is at position t - offs[bi]
    ring = oracle_mod.RingSim(batch, Hkv, d, b, elem)
    for step in range(T):
        t = np.array([step - o for o in offs])
        live = t >= 0
        idx = np.clip(t, 0, None)
        ring.append(K[torch.arange(batch), :, idx], V[torch.arange(batch), :, idx],
                    np.where(live, t, -1))
        if not live.all():
            continue
        q = torch.randn(batch, Hq, d, generator=g).to(dt)
        o_ring = ring.attend(q, t)
        o_full = oracle_mod.attend(q, K, V, s0=0, t=t, b=b)
        assert np.allclose(o_ring, o_full, rtol=1e-12, atol=1e-12)


def test_ring_replay_matches_appends(oracle_mod):
    import torch

    g = torch.Generator().manual_seed(12)
    b, d = 8, 4
    hist = torch.randn(2, 1, b, d, generator=g)
    s0 = np.array([-3, 20])
    a = oracle_mod.RingSim(2, 1, d, b, 4)
    a.replay(hist, hist, s0)
    bsim = oracle_mod.RingSim(2, 1, d, b, 4)
    for j in range(b):
        t = s0 + j
        bsim.append(hist[:, :, j], hist[:, :, j], np.where(t >= 0, t, -1))
    assert np.array_equal(a.k, bsim.k) and np.array_equal(a.tags, bsim.tags)


def test_ring_detects_missing_source(oracle_mod):
    ring = oracle_mod.RingSim(1, 1, 2, 8, 4)
    one = np.ones((1, 1, 2), dtype=np.float32)
    for t in range(10):
        if t != 6:  # position 6 never appended: support of t = 9 is [4, 9]
            ring.append(one, one, t)
    with pytest.raises(oracle_mod.OracleError):
        ring.attend(np.zeros((1, 1, 2)), 9)


# ---------------------------------------------------------- sliding window --


def test_window_score_count_at_8192(oracle_mod):
    """Sec. 3 / App. A.5: SWA-128 uses 1,040,448 scores at n = 8192 (counted by brute force)."""
    g = load("paper_counts.json")
    n, w = g["n"], 128
    assert sum(oracle_mod.window_count(t, w) for t in range(n)) == g["E_SWA"]


@pytest.mark.parametrize("w", [1, 2, 5, 16])
def test_window_predicate(oracle_mod, w):
    for t in range(40):
        for s in range(-2, t + 3):
            assert oracle_mod.in_window(t, s, w) == (max(0, t - w + 1) <= s <= t)


def test_pbb_support_inside_the_window(oracle_mod):
    """App. A.4: with w = b = 2h every PBB source is an SWA source."""
    b = 16
    for t in range(8 * b):
        for s in range(t + 1):
            if oracle_mod.in_support(t, s, b):
                assert oracle_mod.in_window(t, s, b)


def test_window_attention_matches_scipy(oracle_mod):
    from scipy.special import softmax

    rng = np.random.default_rng(21)
    batch, Hq, Hkv, d, w, n = 2, 4, 2, 8, 6, 30
    q, k, v = _rand_problem(rng, batch, Hq, Hkv, d, n)
    ts = np.array([3, 29])
    o = oracle_mod.attend_window(q, k, v, s0=0, t=ts, w=w)
    for bi in range(batch):
        t = int(ts[bi])
        lo = max(0, t - w + 1)
        for j in range(Hq):
            kv = j // (Hq // Hkv)
            z = k[bi, kv, lo:t + 1] @ q[bi, j] / math.sqrt(d)
            ref = softmax(z) @ v[bi, kv, lo:t + 1]
            assert np.allclose(o[bi, j], ref, rtol=1e-13, atol=1e-13)


def test_window_hand_values(oracle_mod):
    """w = 4 at the Fig. 1 size: uniform weights give the mean of the last 4 positions;
    at t = 4 SWA reads {1,2,3,4} (mean 5/2) where PBB reads {2,3,4} (mean 3)."""
    T = 8
    s = np.arange(T, dtype=np.float64)
    v = s.reshape(1, 1, T, 1)
    k = np.zeros_like(v)
    q = np.zeros((1, 1, 1))
    for t in range(T):
        o = oracle_mod.attend_window(q, k, v, s0=0, t=t, w=4)
        lo = max(0, t - 3)
        assert abs(o[0, 0, 0] - (lo + t) / 2) < 1e-12
    assert abs(oracle_mod.attend_window(q, k, v, s0=0, t=4, w=4)[0, 0, 0] - 2.5) < 1e-12
    assert abs(oracle_mod.attend(q, k, v, s0=0, t=4, b=4)[0, 0, 0] - 3.0) < 1e-12


# ------------------------------------------------ whole-sequence forward --


def test_forward_equals_decode_oracle_at_every_position(oracle_mod):
    """The forward at position t is the decode step at t over the same history
    (attend, pinned above): same support, same softmax."""
    rng = np.random.default_rng(31)
    batch, Hq, Hkv, d, b, n = 2, 4, 2, 8, 8, 40
    q = rng.standard_normal((batch, Hq, n, d))
    k = rng.standard_normal((batch, Hkv, n, d))
    v = rng.standard_normal((batch, Hkv, n, d))
    out, _ = oracle_mod.forward(q, k, v, b)
    for t in range(n):
        ref = oracle_mod.attend(q[:, :, t], k[:, :, :t + 1], v[:, :, :t + 1], s0=0, t=t, b=b)
        assert np.array_equal(out[:, :, t], ref), t


def test_forward_matches_scipy_with_log_partition(oracle_mod):
    """scipy softmax and logsumexp over the interval form [a(t), t] (Eq. pbb_relay)."""
    from scipy.special import logsumexp, softmax

    rng = np.random.default_rng(32)
    batch, Hq, Hkv, d, b, n = 1, 6, 3, 4, 6, 31
    q = rng.standard_normal((batch, Hq, n, d))
    k = rng.standard_normal((batch, Hkv, n, d))
    v = rng.standard_normal((batch, Hkv, n, d))
    out, lse = oracle_mod.forward(q, k, v, b)
    for j in range(Hq):
        kv = j // (Hq // Hkv)
        for t in range(n):
            a = interval_start(t, b)
            z = k[0, kv, a:t + 1] @ q[0, j, t] / math.sqrt(d)
            assert np.allclose(out[0, j, t], softmax(z) @ v[0, kv, a:t + 1], rtol=1e-13, atol=1e-13)
            assert abs(lse[0, j, t] - logsumexp(z)) < 1e-12


def test_forward_zero_query_closed_form(oracle_mod):
    """q = 0: every weight is equal, so lse = ln |A(t)| with |A(t)| = h + 1 + (t mod h)
    after the first block (Eq. pbb_cache_support), and out is the support's mean of V."""
    rng = np.random.default_rng(33)
    b, d, n = 16, 3, 100
    h = b // 2
    k = rng.standard_normal((1, 1, n, d))
    v = rng.standard_normal((1, 1, n, d))
    out, lse = oracle_mod.forward(np.zeros((1, 1, n, d)), k, v, b)
    for t in range(n):
        size = t + 1 if t < b else h + 1 + t % h
        assert abs(lse[0, 0, t] - math.log(size)) < 1e-12
        assert np.allclose(out[0, 0, t], v[0, 0, interval_start(t, b):t + 1].mean(axis=0), atol=1e-13)


def test_forward_hand_values(oracle_mod):
    """Hand-derived outputs of the Fig. 1 size (b = 4) for every position of one sequence."""
    g = load("hand_b4.json")
    b, T = g["b"], 12
    s = np.arange(T, dtype=np.float64)
    v = s.reshape(1, 1, T, 1)
    for case, (qv, kv) in {"uniform weights": (0.0, np.zeros_like(s)),
                           "weights 3 and 1": (1.0, np.where(s % 2 == 0, math.log(3.0), 0.0))}.items():
        c = next(c for c in g["cases"] if c["name"] == case)
        out, _ = oracle_mod.forward(np.full((1, 1, T, 1), qv), kv.reshape(1, 1, T, 1), v, b)
        for t in range(T):
            assert abs(out[0, 0, t, 0] - _frac(c["out"][t])) < 1e-12, (case, t)


def test_forward_first_position(oracle_mod):
    """t = 0: the support is {0}: out = v_0 exactly and lse = z_00 = q_0.k_0/sqrt(d)."""
    rng = np.random.default_rng(34)
    q = rng.standard_normal((2, 4, 5, 16))
    k = rng.standard_normal((2, 2, 5, 16))
    v = rng.standard_normal((2, 2, 5, 16))
    out, lse = oracle_mod.forward(q, k, v, 4)
    for j in range(4):
        assert np.array_equal(out[:, j, 0], v[:, j // 2, 0])
        assert np.allclose(lse[:, j, 0], (q[:, j, 0] * k[:, j // 2, 0]).sum(-1) / 4.0, atol=1e-14)


def test_forward_rows_subset(oracle_mod):
    """Requested rows equal the same rows of the full evaluation."""
    rng = np.random.default_rng(35)
    q = rng.standard_normal((2, 4, 20, 8))
    k = rng.standard_normal((2, 1, 20, 8))
    v = rng.standard_normal((2, 1, 20, 8))
    out, lse = oracle_mod.forward(q, k, v, 8)
    rows = np.array([[0, 0, 0], [1, 3, 19], [0, 2, 7], [1, 1, 8]])
    o2, l2 = oracle_mod.forward(q, k, v, 8, rows=rows)
    for i, (bi, j, t) in enumerate(rows):
        assert np.array_equal(o2[i], out[bi, j, t]) and l2[i] == lse[bi, j, t]


# ----------------------------------------------------------------- backward --


def _loss_and_grads(oracle_mod, q, k, v, w_out, b):
    out, _ = oracle_mod.forward(q, k, v, b)
    return float((out * w_out).sum()), oracle_mod.backward(q, k, v, w_out, b)


@pytest.mark.parametrize("b,G", [(4, 1), (4, 2), (6, 3), (8, 2)])
def test_backward_matches_finite_differences(oracle_mod, b, G):
    """Central differences of L = sum(dO * O) through the forward oracle (pinned above)
    against the analytic gradients, for every element of q, k and v."""
    rng = np.random.default_rng(40 + b + G)
    Hkv, n, d = 2, 13, 3
    q = rng.standard_normal((1, Hkv * G, n, d))
    k = rng.standard_normal((1, Hkv, n, d))
    v = rng.standard_normal((1, Hkv, n, d))
    w = rng.standard_normal((1, Hkv * G, n, d))
    _, (dq, dk, dv) = _loss_and_grads(oracle_mod, q, k, v, w, b)
    eps = 1e-6
    for x, g in ((q, dq), (k, dk), (v, dv)):
        num = np.zeros_like(x)
        for idx in np.ndindex(x.shape):
            old = x[idx]
            x[idx] = old + eps
            lp, _ = _loss_and_grads(oracle_mod, q, k, v, w, b)
            x[idx] = old - eps
            lm, _ = _loss_and_grads(oracle_mod, q, k, v, w, b)
            x[idx] = old
            num[idx] = (lp - lm) / (2 * eps)
        assert np.allclose(g, num, rtol=1e-6, atol=1e-7)


def test_backward_key_gradients_sum_to_zero(oracle_mod):
    """A common shift c of every key adds q_t.c/sqrt(d) to all of a row's logits, which the
    softmax ignores: sum_s dk_s = 0 for each (sequence, KV head)."""
    rng = np.random.default_rng(41)
    q = rng.standard_normal((2, 4, 50, 8))
    k = rng.standard_normal((2, 2, 50, 8))
    v = rng.standard_normal((2, 2, 50, 8))
    w = rng.standard_normal((2, 4, 50, 8))
    _, dk, _ = oracle_mod.backward(q, k, v, w, 16)
    assert np.abs(dk.sum(axis=2)).max() < 1e-11


def test_backward_zero_query_closed_form(oracle_mod):
    """q = 0: P_ts = 1/|A(t)| on [a(t), t], so dv_s = sum over t with s in [a(t), t] of dO_t/|A(t)|."""
    rng = np.random.default_rng(42)
    b, n, d = 8, 40, 3
    k = rng.standard_normal((1, 1, n, d))
    v = rng.standard_normal((1, 1, n, d))
    w = rng.standard_normal((1, 1, n, d))
    _, _, dv = oracle_mod.backward(np.zeros((1, 1, n, d)), k, v, w, b)
    ref = np.zeros((n, d))
    for t in range(n):
        a = interval_start(t, b)
        ref[a:t + 1] += w[0, 0, t] / (t + 1 - a)
    assert np.allclose(dv[0, 0], ref, atol=1e-13)


def test_backward_bridge_gradients_reach_exactly_the_bridge_keys(oracle_mod):
    """The paper's multi-block gradient check at B = 8 (h = 4): upstream gradient only on the
    bridge queries 8..11 of block 1. By Eq. (pbb) they attend to the previous block's second
    half (keys 4..7, the bridge) and to their own block up to themselves, so dk and dv are
    nonzero on keys 4..11 (each of them, for generic inputs) and exactly zero on keys 0..3 and
    12 onward; dq is zero outside rows 8..11."""
    rng = np.random.default_rng(43)
    b, n, d = 8, 24, 4
    q = rng.standard_normal((1, 2, n, d))
    k = rng.standard_normal((1, 1, n, d))
    v = rng.standard_normal((1, 1, n, d))
    w = np.zeros((1, 2, n, d))
    w[:, :, 8:12] = rng.standard_normal((1, 2, 4, d))
    dq, dk, dv = oracle_mod.backward(q, k, v, w, b)
    for g in (dk, dv):
        assert np.all(np.abs(g[0, 0, 4:12]).max(axis=-1) > 0)
        assert np.abs(g[0, 0, :4]).max() == 0.0 and np.abs(g[0, 0, 12:]).max() == 0.0
    assert np.abs(dq[0, :, :8]).max() == 0.0 and np.abs(dq[0, :, 12:]).max() == 0.0
    assert np.all(np.abs(dq[0, :, 8:12]).max(axis=-1) > 0)
