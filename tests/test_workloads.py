"""The seeded generator: reproducible, right shapes, right structure."""
import numpy as np
import pytest

from paper_2609_38706_gb300 import workloads as W


def test_reproducible():
    a, b = W.reduced("multi_adapter"), W.reduced("multi_adapter")
    assert np.array_equal(a.batch.tokens, b.batch.tokens)
    assert np.array_equal(a.batch.tok_off, b.batch.tok_off)
    assert np.array_equal(a.filler, b.filler)
    assert a.descriptors == b.descriptors


def test_tiny_shape():
    wl = W.tiny()
    assert wl.batch.R == 8 and wl.batch.n_tokens == 8 * 512 and wl.chunk_tokens == 256
    assert wl.capacity == 64 and wl.target_entries == 16
    assert len({tuple(sorted(d.items())) for d in wl.descriptors}) == 4
    t = wl.batch.tokens.reshape(8, 512)
    assert np.array_equal(t[4], t[0]) and np.array_equal(t[5], t[1])
    assert wl.batch.desc_idx[5] == wl.batch.desc_idx[1] and wl.batch.desc_idx[4] != wl.batch.desc_idx[0]
    d0, d4 = wl.descriptors[wl.batch.desc_idx[0]], wl.descriptors[wl.batch.desc_idx[4]]
    assert [k for k in d0 if d0[k] != d4[k]] == ["adapter_id"]
    assert t.min() >= 0 and t.max() < 32000


def test_filler_distinct_nonzero():
    f = W.filler_keys(5, 20000)
    assert f.shape == (20000, 16)
    assert np.unique(f.view("V16")).size == 20000
    assert f.any(axis=1).all()


def test_multi_adapter_structure():
    wl = W.multi_adapter(R=50, T=4096, capacity_log2=12)
    t = wl.batch.tokens.reshape(50, 4096)
    share = [r for r in range(50) if r % 5 < 2]
    assert all(np.array_equal(t[r, :2048], t[share[0], :2048]) for r in share)
    assert not np.array_equal(t[2, :2048], t[0, :2048])
    assert len(wl.descriptors) == 32 and wl.target_entries == 2048
    assert t.max() < 152064


def test_ragged_has_partial_and_empty():
    wl = W.reduced("multi_adapter")
    lens = np.diff(wl.batch.tok_off)
    assert np.any(lens % 256 != 0) and np.any(lens < 256) and np.any(lens % 256 == 0)
    assert np.any(wl.batch.tok_off[:-1] % 4 != 0)      # unaligned request starts


@pytest.mark.parametrize("D", [1, 4, 16, 64])
def test_sweep_descriptors_distinct(D):
    wl = W.provenance_sweep(D, R=2 * D, T=512, prefix_len=256, capacity_log2=10)
    assert len({tuple(sorted(d.items())) for d in wl.descriptors}) == D
    assert wl.prior.R == D


def test_full_config_sizes_declared():
    # sizes the full configurations promise, without generating them
    import inspect
    assert inspect.signature(W.multi_adapter).parameters["R"].default == 1024
    assert inspect.signature(W.small_block).parameters["R"].default == 16384
    assert inspect.signature(W.long_context).parameters["T"].default == 131072
    assert inspect.signature(W.provenance_sweep).parameters["capacity_log2"].default == 24
