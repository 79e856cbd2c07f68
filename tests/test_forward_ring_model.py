"""Models, on the CPU, of two synchronisation rules of the paired forward kernel: its
per-iteration K/V barrier ring, and which softmax warpgroup frees each K/V stage.

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


# ---- who frees the K/V stages ------------------------------------------------------------
# The paired kernel's softmax warpgroups free the K and V stages: the first thread of item x's
# warpgroup frees K_j and V_{j-1} after seeing x's s_full of tile j when x owns iteration j
# (item B owns its tiles, item A the iterations below B's first tile, all of them without B),
# and V_{nt-1} after x's pv_last when x owns the last iteration. A stage freed twice would let a
# copy overwrite a tile still being read; one never freed stalls the producer. The geometry is
# the kernel's make_pitem, restated.

def support_start(t, h):
    m = t // h
    return h * (m - 1) if m > 0 else 0


def make_pitem(sidx, n, B, QT, NK=128):
    nq = (n + QT - 1) // QT
    nsp = (nq + 1) // 2
    pair = sidx // nsp
    t0 = (sidx - pair * nsp) * 2 * QT
    tlA = min(t0 + QT, n) - 1
    hasB = t0 + QT < n
    tlB = min(t0 + 2 * QT, n) - 1 if hasB else tlA
    h = B // 2
    loA = support_start(t0, h)
    loB = support_start(t0 + QT, h) if hasB else loA
    return {"hasB": hasB, "nt": (tlB - loA + NK) // NK, "ntA": (tlA - loA + NK) // NK,
            "jB0": (loB - loA) // NK}


def check_item_releases(it):
    nt, hasB = it["nt"], it["hasB"]
    jb = [0, it["jB0"] if hasB else nt]
    je = [it["ntA"], nt]
    # the issuing thread's commits, in order, per iteration j = 0 .. nt
    last_commit = {}
    for j in range(nt + 1):
        for x in (0, 1):
            sk = jb[x] <= j < je[x]
            pv = j >= jb[x] + 1 and j - 1 < je[x]
            if sk:
                last_commit[j] = ("s_full", x)
            elif pv:
                last_commit[j] = ("pv_last", x)
    assert set(last_commit) == set(range(nt + 1)), "an iteration without products"
    freed = {"k": [], "v": []}
    for x in (0, 1):
        if x == 1 and not hasB:
            continue
        jown = nt if x == 1 else (it["jB0"] if hasB else nt)
        for j in range(jb[x], je[x]):
            if j < jown:  # after x's s_full of tile j
                assert last_commit[j] == ("s_full", x), (it, j, x)
                freed["k"].append(j)
                if j >= 1:
                    freed["v"].append(j - 1)
        if x == 1 or not hasB:  # after x's pv_last, the item's last P.V
            assert last_commit[nt] == ("pv_last", x), (it, x)
            freed["v"].append(nt - 1)
    assert sorted(freed["k"]) == list(range(nt)), (it, freed)
    assert sorted(freed["v"]) == list(range(nt)), (it, freed)


@pytest.mark.parametrize("B", [512, 768, 1024, 2048, 4096])
@pytest.mark.parametrize("group", [1, 2, 4, 8])
def test_every_stage_is_freed_once_by_the_last_reader(B, group):
    QT = 128 // group
    for n in (1, 31, 32, 33, 63, 64, 65, 100, 777, 2 * B + 5, 3 * B):
        nq = (n + QT - 1) // QT
        for sidx in range((nq + 1) // 2):  # one (sequence, KV head): the items repeat per pair
            check_item_releases(make_pitem(sidx, n, B, QT))
