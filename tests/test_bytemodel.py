"""CPU checks of the byte/FLOP model the benchmark's roofline uses: its support
sizes are pinned to the oracle's brute-force counts and to the paper's score
budgets, and its byte count to a by-hand tally of one sequence."""
import json
import os

import numpy as np
import pytest

from paper_2606_02680_gb300 import bytemodel

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_support_sizes_match_the_oracle(oracle_mod):
    for B in (2, 8, 96, 128):
        t = np.arange(6 * B)
        assert list(bytemodel.support_size(t, B)) == [oracle_mod.support_count(int(x), B) for x in t]
        for w in (1, B // 2, B):
            assert list(bytemodel.support_size(t, B, w)) == [oracle_mod.window_count(int(x), w) for x in t]


def test_score_budgets_at_8192():
    g = json.load(open(os.path.join(GOLDEN, "paper_counts.json")))
    t = np.arange(g["n"])
    assert int(bytemodel.support_size(t, g["b"]).sum()) == g["E_PBB"]
    assert int(bytemodel.support_size(t, g["b"], g["b"]).sum()) == g["E_SWA"]
    assert bytemodel.mean_support(g["b"]) == g["phase_mean_support_h64"]


@pytest.mark.parametrize("window", [None, 4096])
def test_step_bytes_by_hand(window):
    """One bf16 sequence, Hq 32, Hkv 8, d 128, B 4096, t = 3*4096 + 5 (a bridge phase):
    PBB reads 2048 + 5 ring keys, the window 4095."""
    t, Hq, Hkv, d, e = 3 * 4096 + 5, 32, 8, 128, 2
    ring_keys = 2048 + 5 if window is None else 4095
    want = Hkv * d * e * (2 * ring_keys + 2 + 2) + Hq * d * e + Hq * d * 4 + 4
    assert bytemodel.step_bytes([t], Hq, Hkv, d, 4096, e, window) == want
    assert bytemodel.step_flops([t], Hq, d, 4096, window) == 4 * d * Hq * (ring_keys + 1)
