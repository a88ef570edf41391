"""Host-side logic of the step loop that needs no GPU: how a batch is cut
into sub-batches for the pipelined loop."""
import pytest

from paper_2502_17139_gb300.step import sub_batch_slices


@pytest.mark.parametrize("B", [1, 2, 9, 16, 32, 33, 1000])
def test_sub_batches_partition_the_batch(B):
    for n in range(1, min(B, 12) + 1):
        sl = sub_batch_slices(B, n)
        assert len(sl) == n
        assert sl[0].start == 0 and sl[-1].stop == B
        assert all(a.stop == b.start for a, b in zip(sl, sl[1:]))
        sizes = [s.stop - s.start for s in sl]
        assert max(sizes) - min(sizes) <= 1 and min(sizes) >= 1


def test_sub_batch_bounds():
    assert [(s.start, s.stop) for s in sub_batch_slices(32, 2)] == [(0, 16), (16, 32)]
    assert [(s.start, s.stop) for s in sub_batch_slices(32, 3)] == [(0, 10), (10, 21), (21, 32)]
    for bad in (0, 33):
        with pytest.raises(ValueError):
            sub_batch_slices(32, bad)
