"""GPU parity of the store-side omission test: worker A's keys stored in a
table (slot = page index), worker B's keys looked up in it, the joined pages
compared by pk_compare_pages; verdicts and counts equal the oracle's, for
complete and leave-one-out bindings.  Plus the comparison kernel's own edge
cases against the oracle's compare_pages."""
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


def gpu_check(case):
    from paper_2609_38706_gb300 import pk
    from paper_2609_38706_gb300.service import KeyTable
    b, C = case.batch, case.chunk_tokens
    kt = KeyTable(C, 12)
    _, ka = kt.derive(b.tokens, b.tok_off, b.desc_idx, kt.digests([case.bound_a]))
    _, kb = kt.derive(b.tokens, b.tok_off, b.desc_idx, kt.digests([case.bound_b]))
    n = ka.shape[0]
    kt.store(ka, np.arange(n, dtype=np.uint32))                      # reference worker's keys -> page index
    one = torch.tensor([0, n], dtype=torch.int64, device="cuda")
    _, slots = kt.lookup(kb, one)
    kt.check("join")
    verdict = torch.empty(n, dtype=torch.int32, device="cuda")
    counts = torch.zeros(3, dtype=torch.int64, device="cuda")
    pk.pk_compare_pages(slots, torch.from_numpy(case.pages_b).cuda(), torch.from_numpy(case.pages_a).cuda(),
                        verdict, counts, kt.status, kt.stream)
    kt.check("compare")
    out = verdict.cpu().numpy(), counts.cpu().numpy(), ka.cpu().numpy(), kb.cpu().numpy()
    kt.close()
    return out


@pytest.mark.parametrize("varied,omit", [("weight_version", None), ("weight_version", "weight_version"),
                                         ("kv_format", "kv_format"), ("adapter_id", "adapter_id"),
                                         ("salt", "salt"), ("adapter_id", "salt")])
def test_omission_check_matches_oracle(varied, omit):
    case = W.omission_case(varied, omit)
    verdict, counts, ka, kb = gpu_check(case)
    rv, rc = O.omission_check(ka, case.pages_a, kb, case.pages_b)
    assert np.array_equal(verdict, rv) and np.array_equal(counts, rc)


def test_compare_pages_edges():
    from paper_2609_38706_gb300 import pk
    rng = np.random.default_rng(3)
    n, n_ref, P = 300, 40, 48 * 16
    ref = rng.integers(0, 256, (n_ref, P), dtype=np.uint8)
    slots = rng.integers(0, n_ref, n).astype(np.uint32)
    slots[::7] = O.NO_SLOT
    pages = ref[np.where(slots == O.NO_SLOT, 0, slots)].copy()
    flip = rng.choice(n, 50, replace=False)
    pages[flip, rng.integers(0, P, 50)] ^= 0x10                      # a difference anywhere in the page
    pages[5, P - 1] ^= 1                                             # ... including the last byte
    rv, rc = O.compare_pages(slots, pages, ref)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    verdict = torch.empty(n, dtype=torch.int32, device="cuda")
    counts = torch.zeros(3, dtype=torch.int64, device="cuda")
    pk.pk_compare_pages(torch.from_numpy(slots.view(np.int32)).cuda(), torch.from_numpy(pages).cuda(),
                        torch.from_numpy(ref).cuda(), verdict, counts, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert np.array_equal(verdict.cpu().numpy(), rv) and np.array_equal(counts.cpu().numpy(), rc)
    # a slot naming no reference page: reported, and read as absent
    bad = slots.copy()
    bad[3] = n_ref
    verdict.zero_()
    counts.zero_()
    pk.pk_compare_pages(torch.from_numpy(bad.view(np.int32)).cuda(), torch.from_numpy(pages).cuda(),
                        torch.from_numpy(ref).cuda(), verdict, counts, status)
    torch.cuda.synchronize()
    assert int(status.item()) == pk.PK_ERR_ARG and int(verdict[3].item()) == O.PAGE_ABSENT
    # host checks: page size not a multiple of 16
    with pytest.raises(pk.PKError):
        pk.pk_compare_pages(torch.from_numpy(slots.view(np.int32)).cuda(),
                            torch.zeros((n, 24), dtype=torch.uint8, device="cuda"),
                            torch.zeros((n_ref, 24), dtype=torch.uint8, device="cuda"), verdict, counts, status)
