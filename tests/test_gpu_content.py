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
