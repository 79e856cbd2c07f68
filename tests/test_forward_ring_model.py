"""A model, on the CPU, of the paired forward kernel's per-iteration K/V barrier ring.

Iteration i of the issuing thread (S on K_j, P.V on V_{j-1}; j = 0 .. nt per item) waits on
slot i mod R of a ring of mbarriers. The K and the V producer each arrive on that slot once per
iteration: with a copy's bytes, or without a copy where they have none (K at j = nt, V at
j = 0). Before copying tile t into its ring of S stages, a producer waits for tile t - S to be
freed, which happens some time after the issuing thread has passed the iteration that read it.
A slot may take arrivals for iteration i only once the issuing thread has passed iteration
i - R, else two phases of the slot overlap. The kernel sizes the ring as
R = 2 max(S_K, S_V) + 2. This test drives the protocol under random interleavings, random
copy latencies and random release delays, and checks that rule (and that the previous fixed
R = 8 fails with the four K and four V stages of d = 64).
"""
import random

import pytest


def iterations(nts):
    """Per iteration: (K tile or None, V tile or None), over items with nt K/V tiles each."""
    out, t = [], 0
    for nt in nts:
        for j in range(nt + 1):
            out.append((t + j if j < nt else None, t + j - 1 if j >= 1 else None))
        t += nt
    return out


def simulate(nts, sk, sv, ring, rng):
    """Runs the protocol to the end; returns the number of arrivals that landed on a slot whose
    previous iteration the issuing thread had not yet passed."""
    its = iterations(nts)
    n = len(its)
    arrivals = [0] * n
    in_flight = [0] * n              # copies not yet landed, per iteration
    landing = []                     # (iteration) of copies in flight
    freed = {"k": set(), "v": set()}
    to_free = []                     # (kind, tile) readable by the issuing thread already
    pos = {"k": 0, "v": 0}           # next iteration of each producer
    copies = {"k": 0, "v": 0}        # tiles copied so far
    passed = 0                       # iterations the issuing thread has passed
    stages = {"k": sk, "v": sv}
    violations = 0
    while passed < n:
        moves = []
        for kind in ("k", "v"):
            i = pos[kind]
            if i < n:
                tile = its[i][0 if kind == "k" else 1]
                if tile is None or copies[kind] < stages[kind] or (copies[kind] - stages[kind]) in freed[kind]:
                    moves.append(("produce", kind))
        if landing:
            moves.append(("land", None))
        if to_free:
            moves.append(("free", None))
        if arrivals[passed] == 2 and in_flight[passed] == 0:
            moves.append(("consume", None))
        assert moves, "deadlock"
        what, kind = rng.choice(moves)
        if what == "produce":
            i = pos[kind]
            if i >= ring and passed <= i - ring:
                violations += 1
            arrivals[i] += 1
            if its[i][0 if kind == "k" else 1] is not None:
                in_flight[i] += 1
                landing.append(i)
                copies[kind] += 1
            pos[kind] += 1
        elif what == "land":
            i = landing.pop(rng.randrange(len(landing)))
            in_flight[i] -= 1
        elif what == "free":
            kind, tile = to_free.pop(rng.randrange(len(to_free)))
            freed[kind].add(tile)
        else:
            k_tile, v_tile = its[passed]
            if k_tile is not None:
                to_free.append(("k", k_tile))
            if v_tile is not None:
                to_free.append(("v", v_tile))
            passed += 1
    return violations


def kernel_ring(sk, sv):
    """The kernel's rule (PairCfg::KVR)."""
    return 2 * max(sk, sv) + 2


ITEM_MIXES = {
    "one_tile": lambda rng: [1] * 40,
    "short": lambda rng: [rng.randint(1, 3) for _ in range(30)],
    "mixed": lambda rng: [rng.choice([1, 1, 2, 5, 16]) for _ in range(20)],
}


@pytest.mark.parametrize("sk,sv", [(3, 2), (4, 4)])  # d = 128 and d = 64
@pytest.mark.parametrize("mix", list(ITEM_MIXES))
def test_kernel_ring_never_overlaps_phases(sk, sv, mix):
    rng = random.Random(f"{sk}{sv}{mix}")
    for _ in range(300):
        assert simulate(ITEM_MIXES[mix](rng), sk, sv, kernel_ring(sk, sv), rng) == 0


def test_the_model_finds_the_overlap_of_a_short_ring():
    """With four K and four V stages a producer arrives up to 2 S = 8 iterations past the last
    one the issuing thread has passed: a ring of 8 (the kernel's first sizing) lets some
    schedule overlap two phases, while 2 S + 1 = 9, one slot fewer than the kernel keeps, does
    not."""
    rng = random.Random(7)
    assert sum(simulate([1] * 40, 4, 4, 8, rng) for _ in range(300)) > 0
    assert sum(simulate([1] * 40, 4, 4, 9, rng) for _ in range(300)) == 0
