"""GPU parity of the content identity: pk_content_digest (the SHA-256 tree on
the device) against the oracle's tree, bit-exact, across sizes that hit every
edge of the tree (empty, partial 16-byte tails, one block, block boundaries,
two and three levels), and an adapter's identity end to end."""
import numpy as np
import pytest
import torch

import oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no GPU")


def gpu_top(data: np.ndarray) -> bytes:
    from paper_2609_38706_gb300 import pk
    d = torch.from_numpy(data).cuda() if data.size else torch.zeros(16, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(pk.pk_content_scratch_bytes(data.size), dtype=torch.uint8, device="cuda")
    top = torch.empty(32, dtype=torch.uint8, device="cuda")
    pk.pk_content_digest(d[: data.size], scratch, top)
    return bytes(top.cpu().numpy())


@pytest.mark.parametrize("n", [0, 1, 15, 16, 17, 1023, 1024, 1025, 4099, 65536, 33 * 1024 + 1, (1 << 20) + 5])
def test_tree_top_bit_exact(n):
    data = np.random.default_rng(n).integers(0, 256, n, dtype=np.uint8)
    assert gpu_top(data) == O.content_digest(data.tobytes())


def test_large_buffer_against_the_oracle():
    data = np.random.default_rng(77).integers(0, 256, 9 * (1 << 20) + 333, dtype=np.uint8)   # four levels
    assert gpu_top(data) == O.content_digest(data.tobytes())


def test_level_of_many_blocks_against_the_oracle():
    """96 MiB: a first tree level of 98,305 blocks, enough warps per SM sub-partition for the multiply-add
    round form (every addition on the FMA pipe), bit-exact like the compiler's form."""
    data = np.random.default_rng(96).integers(0, 256, 96 * (1 << 20) + 5, dtype=np.uint8)
    assert gpu_top(data) == O.content_digest(data.tobytes())


def test_adapter_identity_end_to_end():
    from paper_2609_38706_gb300 import pk
    rng = np.random.default_rng(8)
    tensors = {f"layers.{i}.{p}": rng.standard_normal((64, 16 * (i + 1))).astype(np.float16)
               for i in range(3) for p in ("lora_A", "lora_B")}
    ids, rids = [], []
    for name in sorted(tensors):
        t = tensors[name]
        raw = t.view(np.uint8).reshape(-1)
        top = gpu_top(raw)
        ids.append(pk.pk_tensor_identity(name, "fp16", t.shape, raw.size, top))
        rids.append(O.tensor_identity(name, "fp16", t.shape, raw.size, O.content_digest(raw.tobytes())))
    cfg = ["r=16", "lora_alpha=32", "target_modules=q_proj,v_proj"]
    assert pk.pk_adapter_identity(ids, cfg) == O.adapter_identity(rids, cfg)


def test_host_argument_errors():
    from paper_2609_38706_gb300 import pk
    d = torch.zeros(4096 + 16, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(pk.pk_content_scratch_bytes(4096), dtype=torch.uint8, device="cuda")
    top = torch.empty(32, dtype=torch.uint8, device="cuda")
    with pytest.raises(pk.PKError):   # misaligned source
        pk.pk_content_digest(d[1:4097], scratch, top)
    with pytest.raises(pk.PKError):   # scratch too small
        pk.pk_content_digest(d[:4096], scratch[:32], top)


def gpu_tops(datas):
    from paper_2609_38706_gb300 import pk
    ts = [torch.from_numpy(d).cuda() if d.size else torch.zeros(0, dtype=torch.uint8, device="cuda") for d in datas]
    scratch = torch.empty(max(pk.pk_content_scratch_bytes_batch([d.size for d in datas]), 16), dtype=torch.uint8,
                          device="cuda")
    tops = torch.empty((max(len(datas), 1), 32), dtype=torch.uint8, device="cuda")
    pk.pk_content_digests(ts, scratch, tops)
    return [bytes(r) for r in tops.cpu().numpy()[: len(datas)]]


def test_batch_of_mixed_sizes():
    """Buffers that end at different tree levels in one call (empty, one block,
    two, three and four levels): each top equals the oracle's and the one-buffer
    call's."""
    rng = np.random.default_rng(21)
    sizes = [0, 1, 1024, 1025, 65536 + 3, 33 * 1024, 0, 9 * (1 << 20) + 333, 17, (1 << 20) + 5]
    datas = [rng.integers(0, 256, n, dtype=np.uint8) for n in sizes]
    got = gpu_tops(datas)
    for d, g in zip(datas, got):
        assert g == O.content_digest(d.tobytes())
        assert g == gpu_top(d)


def test_batch_larger_than_one_launch():
    """300 buffers: more than one launch's 128 segments per level."""
    rng = np.random.default_rng(22)
    sizes = rng.integers(0, 40_000, 300)
    sizes[::37] = 0
    datas = [rng.integers(0, 256, int(n), dtype=np.uint8) for n in sizes]
    got = gpu_tops(datas)
    assert got == [O.content_digest(d.tobytes()) for d in datas]


def test_batch_adapter_identity():
    from paper_2609_38706_gb300 import pk
    rng = np.random.default_rng(23)
    tensors = {f"layers.{i}.{p}": rng.standard_normal((128, 8 * (i + 1))).astype(np.float16)
               for i in range(24) for p in ("lora_A", "lora_B")}
    names = sorted(tensors)
    raws = [tensors[k].view(np.uint8).reshape(-1) for k in names]
    tops = gpu_tops(raws)
    ids = [pk.pk_tensor_identity(k, "fp16", tensors[k].shape, r.size, t) for k, r, t in zip(names, raws, tops)]
    rids = [O.tensor_identity(k, "fp16", tensors[k].shape, r.size, O.content_digest(r.tobytes()))
            for k, r in zip(names, raws)]
    assert pk.pk_adapter_identity(ids, ["r=8"]) == O.adapter_identity(rids, ["r=8"])


def test_batch_host_errors():
    import ctypes
    from paper_2609_38706_gb300 import pk
    L = pk.lib()
    d = torch.zeros(4096 + 16, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(1 << 16, dtype=torch.uint8, device="cuda")
    tops = torch.empty((2, 32), dtype=torch.uint8, device="cuda")
    ptrs = (ctypes.c_void_p * 2)(d.data_ptr(), d.data_ptr() + 8)  # the second misaligned
    sizes = (ctypes.c_uint64 * 2)(4096, 4096)
    assert L.pk_content_digests(ptrs, sizes, 2, scratch.data_ptr(), scratch.numel(), tops.data_ptr(), None) == pk.PK_ERR_ARG
    ptrs = (ctypes.c_void_p * 2)(d.data_ptr(), d.data_ptr())
    assert L.pk_content_digests(ptrs, sizes, 2, scratch.data_ptr(), 64, tops.data_ptr(), None) == pk.PK_ERR_ARG
    assert L.pk_content_digests(None, None, 0, None, 0, None, None) == pk.PK_OK
