"""Slice samples of the synthetic workloads: a sample holds the same shapes
and the same values as those slices of the whole workload (what `bench.py
--slices N` and the oracle's bounded samples rely on)."""
import numpy as np

from paper_2002_07062_gb300 import workload


def test_prefix_sample_of_the_ragged_workload_is_its_first_slices():
    w = workload.config(4)
    n = 20
    s = workload.slice_sample(w, list(range(n)))
    assert np.array_equal(s.rows, w.rows[:n]) and np.array_equal(s.cols, w.cols[:n])
    assert np.array_equal(s.offsets, w.offsets[:n])
    # the whole workload's values start with these slices: its first elements
    head = workload.fill_normal(s.numel, w.dtype, w.seed, w.sigma)
    assert np.array_equal(s.x.view(np.uint32), head.view(np.uint32))


def test_any_sample_matches_the_materialized_workload():
    for dtype in (workload.F32, workload.BF16):
        w = workload.ragged("small ragged", dtype, 30, 2.0, 0x51CE + dtype, row_steps=4,
                            col_steps=8).materialize()
        pick = [29, 3, 17, 0, 8]
        s = workload.slice_sample(w, pick)
        word = np.uint32 if dtype == workload.F32 else np.uint16
        for j, k in enumerate(pick):
            n = int(w.rows[k]) * int(w.cols[k])
            got = s.x[s.offsets[j]:s.offsets[j] + n].view(word)
            want = w.x[w.offsets[k]:w.offsets[k] + n].view(word)
            assert s.rows[j] == w.rows[k] and s.cols[j] == w.cols[k]
            assert np.array_equal(got, want), (dtype, k)
        assert s.offsets[0] == 0 and s.numel == sum(int(w.rows[k]) * int(w.cols[k]) for k in pick)
