"""Property tests of the host planners on random ragged layouts (CPU, no
device): the chunk table (lamb_layout_chunks), the shard ranges cut from it
(lamb_layout_shard) and the on-chip rounds (lamb_layout_rounds), each checked
against the rule include/lamb.h states for it."""
import numpy as np
import pytest

pytest.importorskip("hypothesis")
from hypothesis import HealthCheck, given, settings  # noqa: E402
from hypothesis import strategies as st  # noqa: E402

from paper_1904_00962_gb300 import binding as B  # noqa: E402
from paper_1904_00962_gb300 import build as build_mod  # noqa: E402
from test_host_abi import _check_rounds  # noqa: E402

SETTINGS = settings(max_examples=150, deadline=None,
                    suppress_health_check=[HealthCheck.too_slow])

# tensor sizes: empty, tiny, around a row or chunk boundary, and large
SIZE = st.one_of(st.integers(0, 4), st.integers(0, 300),
                 st.integers(1000, 70000), st.integers(0, 400000))
SIZES = st.lists(SIZE, min_size=1, max_size=40)
CHUNK = st.sampled_from([1024, 2048, 4096, 16384])
TAIL = st.sampled_from([0, 1, 3000, 50000, 10 ** 9])


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build_mod.build()
    B.load()


def _positions(sizes, t, o):
    starts = np.concatenate([[0], np.cumsum(sizes, dtype=np.int64)[:-1]])
    return starts[t] + o


def _tail_allowed(chunk, tail):
    """A tail of short chunks needs chunks at least that long."""
    return tail == 0 or chunk >= B.LAMB_TAIL_CHUNK_ELEMS


@SETTINGS
@given(sizes=SIZES, chunk=CHUNK, tail=TAIL)
def test_chunks_tile_every_tensor_in_order(sizes, chunk, tail):
    if not _tail_allowed(chunk, tail):
        with pytest.raises(B.LambError) as ei:
            B.lamb_layout_chunks(sizes, chunk, tail)
        assert ei.value.status == B.LAMB_ERR_INVALID_ARG
        return
    t, o, ln = B.lamb_layout_chunks(sizes, chunk, tail)
    total = sum(sizes)
    assert int(ln.sum()) == total
    assert np.all(ln >= 1) and np.all(ln <= chunk)
    assert np.all(np.diff(t) >= 0)
    assert np.all(o % 1024 == 0)
    pos = _positions(sizes, t, o)
    assert np.all(np.diff(pos) > 0)
    for k, s in enumerate(sizes):
        sel = t == k
        if s == 0:
            assert not sel.any()
            continue
        offs, lens = o[sel], ln[sel]
        assert offs[0] == 0 and offs[-1] + lens[-1] == s
        np.testing.assert_array_equal(offs[1:], offs[:-1] + lens[:-1])
    short = B.LAMB_TAIL_CHUNK_ELEMS
    in_tail = ((pos < tail) | (pos + chunk > total - tail)) if tail else \
        np.zeros(len(pos), bool)
    assert np.all(ln[in_tail] <= short)
    ends = o + ln == np.asarray(sizes, dtype=np.int64)[t]
    assert np.all((ln[~in_tail] == chunk) | ends[~in_tail])


@SETTINGS
@given(sizes=SIZES, chunk=CHUNK, tail=TAIL, world=st.integers(1, 9))
def test_shards_split_the_chunk_table_by_elements(sizes, chunk, tail, world):
    if not _tail_allowed(chunk, tail):
        with pytest.raises(B.LambError):
            B.lamb_layout_shard(sizes, world, 0, chunk, tail)
        return
    t, o, ln = B.lamb_layout_chunks(sizes, chunk, tail)
    pos = _positions(sizes, t, o)
    total = sum(sizes)
    ranges = [B.lamb_layout_shard(sizes, world, r, chunk, tail)
              for r in range(world)]
    assert ranges[0][0] == 0 and ranges[-1][1] == len(t)
    for (b0, e0), (b1, _) in zip(ranges, ranges[1:]):
        assert e0 == b1
    for r, (b, e) in enumerate(ranges):
        assert 0 <= b <= e <= len(t)
        lo, hi = total * r // world, total * (r + 1) // world
        inside = (pos >= lo) & (pos < hi)
        np.testing.assert_array_equal(np.flatnonzero(inside),
                                      np.arange(b, e))
        # a rank holds its share of the elements give or take one chunk
        assert abs(int(ln[b:e].sum()) - total / world) <= chunk + 1


@SETTINGS
@given(sizes=st.lists(SIZE, min_size=1, max_size=60),
       grid=st.integers(1, 40), rpc=st.integers(1, 224))
def test_rounds_hold_whole_tensors(sizes, grid, rpc):
    _check_rounds(sizes, grid, rpc)
