"""The planted-attention generator of the homogeneous SnapKV 8K workload,
checked with the statistic the paper uses to show that layers differ (Sec. 1,
Fig. 1): the size of the smallest set of positions that covers 90% of the
head-averaged observation-window attention.

The workload plants, in each of the 32 layers, a support of s_l positions
(16 at the first layer to 1600 at the last) that should carry the window
attention.  The oracle computes the window attention of every layer; the
statistic of each layer must lie within a factor of 2 of s_l, and across
layers it must spread over at least 50x (the paper's layers span about two
orders of magnitude).  Heads 0 and H_kv-1 of every layer are averaged (the
planted direction differs per head, the planted set does not).  CPU only.
"""
import numpy as np

from paper_2606_15157_gb300 import inputs as gen


def support90(a: np.ndarray) -> int:
    """Smallest number of positions whose attention mass reaches 90% of the total."""
    srt = np.sort(a)[::-1]
    c = np.cumsum(srt) / srt.sum()
    return int(np.searchsorted(c, 0.9 - 1e-12) + 1)  # tolerance for the rounding of cumsum


def test_support90_hand_cases():
    assert support90(np.array([0.9, 0.05, 0.05])) == 1
    assert support90(np.array([0.5, 0.3, 0.1, 0.1])) == 3
    assert support90(np.full(10, 0.1)) == 9


def test_planted_support_matches_recipe(orc):
    wl = gen.config_homog8k(seed=0)
    n = int(wl.lens[0])
    pos = np.arange(n, dtype=np.int64)
    sup = []
    for l in range(wl.L):
        a = np.zeros(n)
        for h in (0, wl.H_kv - 1):
            K = gen.k_rows(wl, l, 0, h, pos)
            Q = gen.q_group(wl, l, 0, h)
            a += orc.window_scores(K, Q, n, wl.W)
        m = support90(a)
        s_l = int(wl.plant["size"][l])
        assert s_l / 2 <= m <= 2 * s_l, (l, s_l, m)
        sup.append(m)
    assert max(sup) / min(sup) >= 50
