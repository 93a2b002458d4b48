"""GPU parity of pk_key_strings (Sec. 5.3, connector integration) against the
oracle's key_strings: every byte of every row, for row widths and prefix
lengths at the limits, batch sizes that leave a ragged last tile, and the key
batch of a full workload."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_38706_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no GPU")


def gpu_rows(keys_np, prefix, width, n=None):
    from paper_2609_38706_gb300 import pk
    keys = torch.from_numpy(np.ascontiguousarray(keys_np)).cuda()
    n = keys.shape[0] if n is None else n
    out = torch.full((max(n, 1), width), 0xA5, dtype=torch.uint8, device="cuda")  # poisoned
    pk.pk_key_strings(keys, prefix, width, out, n=n)
    torch.cuda.synchronize()
    return out.cpu().numpy()[:n], out


@pytest.mark.parametrize("n", [0, 1, 7, 255, 256, 257, 1000, 4099])
@pytest.mark.parametrize("prefix,width", [(b"", 22), (b"vllm@tag@1@0@", 150), (b"x" * 234, 256), (b"ab", 33)])
def test_rows_bit_exact(n, prefix, width):
    rng = np.random.default_rng(n * 7 + width)
    keys = rng.integers(0, 256, (max(n, 1), 32), dtype=np.uint8)
    keys[0, :16] = 0 if n else keys[0, :16]          # the all-zero prefix encodes too
    if n > 2:
        keys[1, :16] = 0xFF
    got, _ = gpu_rows(keys, prefix, width, n)
    want = O.key_strings(keys[:n], prefix, width)
    assert np.array_equal(got, want)


def test_writes_nothing_past_the_rows():
    rng = np.random.default_rng(9)
    keys = rng.integers(0, 256, (300, 32), dtype=np.uint8)
    from paper_2609_38706_gb300 import pk
    k = torch.from_numpy(keys).cuda()
    buf = torch.full((301 * 150 + 64,), 0x5A, dtype=torch.uint8, device="cuda")
    pk.pk_key_strings(k, b"p@", 150, buf, n=299)
    torch.cuda.synchronize()
    b = buf.cpu().numpy()
    assert np.array_equal(b[: 299 * 150].reshape(299, 150), O.key_strings(keys[:299], b"p@", 150))
    assert (b[299 * 150:] == 0x5A).all()


@pytest.mark.parametrize("name", ["multi_adapter", "long_context"])
def test_workload_keys(name):
    """The keys of a derived batch (reduced size: every row compared; full
    size: a seeded sample of rows compared)."""
    from paper_2609_38706_gb300.service import KeyTable
    wl = W.reduced(name)
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    d = kt.digests(wl.descriptors)
    key_off, keys = kt.derive(wl.batch.tokens, wl.batch.tok_off, wl.batch.desc_idx, d)
    N = int(key_off[-1])
    prefix = ("vllm@" + O.model_tag(wl.descriptors[0]) + "@1@0@").encode()
    from paper_2609_38706_gb300 import pk
    out = torch.empty((N, 150), dtype=torch.uint8, device="cuda")
    pk.pk_key_strings(keys, prefix, 150, out, n=N)
    torch.cuda.synchronize()
    want = O.key_strings(keys.cpu().numpy()[:N], prefix, 150)
    assert np.array_equal(out.cpu().numpy(), want)
    kt.close()


@pytest.mark.slow
def test_full_multi_adapter_sampled():
    from paper_2609_38706_gb300 import pk
    from paper_2609_38706_gb300.service import KeyTable
    wl = W.FULL_CONFIGS["multi_adapter"]()
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    d = kt.digests(wl.descriptors)
    key_off, keys = kt.derive(wl.batch.tokens, wl.batch.tok_off, wl.batch.desc_idx, d)
    N = int(key_off[-1])
    out = torch.empty((N, 150), dtype=torch.uint8, device="cuda")
    pk.pk_key_strings(keys, b"vllm@" + b"T" * 22 + b"@1@0@", 150, out, n=N)
    torch.cuda.synchronize()
    rng = np.random.default_rng(11)
    idx = np.unique(np.concatenate([rng.integers(0, N, 4000), [0, N - 1]]))
    kh = keys[torch.from_numpy(idx).cuda()].cpu().numpy()
    want = O.key_strings(kh, b"vllm@" + b"T" * 22 + b"@1@0@", 150)
    assert np.array_equal(out[torch.from_numpy(idx).cuda()].cpu().numpy(), want)
    kt.close()


@pytest.mark.parametrize("n,width,prefix", [(200_003, 150, b"vllm@" + b"M" * 22 + b"@1@0@"), (100_001, 256, b"q" * 200),
                                            (81_920, 22, b"")])
def test_several_tiles_per_block(n, width, prefix):
    """More rows than the resident CTAs hold at once (each CTA takes several
    tiles, alternating its two shared-memory tiles): every row compared."""
    rng = np.random.default_rng(n)
    keys = rng.integers(0, 256, (n, 32), dtype=np.uint8)
    got, _ = gpu_rows(keys, prefix, width)
    want = O.key_strings(keys, prefix, width)
    bad = np.nonzero((got != want).any(axis=1))[0]
    assert bad.size == 0, f"{bad.size} rows differ, first {bad[:5]}"
