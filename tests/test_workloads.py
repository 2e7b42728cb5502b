"""The mixed adaptive generator (workloads.adaptive_mixed): its coherent
windows must score high on Eq. redundancy and the others low, so that the
router's decision at rho = 4 and 8 follows the generator's choice."""
import numpy as np

import oracle as O
import workloads as WL


def test_coherent_windows_score_high_and_others_low():
    w = WL.scaled(WL.WORKLOADS["adaptive_mixed"], N=8192, d=256, batch=1)
    nc = w.N - w.preserve_first - w.preserve_last
    for index in (1, 9):
        X = WL.make_prompt(w, index=index).x_f64()
        coherent = {a for a, _, _ in WL.coherent_windows(w, index=index)}
        for s0, e0 in O.window_bounds(nc, w.window):
            sc = O.redundancy_score(X[s0:e0])
            if s0 in coherent:
                assert sc > 0.75 > O.tau_schedule(4.0)
            else:
                assert sc < 0.2 < O.tau_schedule(8.0)


def test_coherent_windows_are_reproducible_and_seeded():
    w = WL.WORKLOADS["adaptive_mixed"]
    a = WL.coherent_windows(w, index=3)
    b = WL.coherent_windows(w, index=3)
    assert [x[:2] for x in a] == [x[:2] for x in b]
    assert all(np.array_equal(x[2], y[2]) for x, y in zip(a, b))
    frac = np.mean([len(WL.coherent_windows(w, index=i)) / 8 for i in range(64)])
    assert 0.35 < frac < 0.65
