"""The allocation-free top-q entry point (scoot_select_topq_static).

It serves callers that cannot allocate device memory when they select, so
it keeps its partial results in a fixed device array instead of a context
workspace.  Its picks must equal scoot_select_topq's exactly, on calls made
one after the other on the same stream (the second call sees the array as
the first left it), and the oracle's selection.  This file is collected last so that a failure here does
not hide any other test."""
import numpy as np
import pytest

import oracle as O
from workloads import Stream

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def S():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2408_04323_gb300 as pkg
    pkg.build()
    from paper_2408_04323_gb300 import scoot
    return scoot


def _case(seed, n):
    st = Stream(seed, "no-alloc")
    acq = np.round(st.normal(n) * 4.0).astype(np.float32) / 4  # ties
    acq[st.uniform(n) < 0.05] = -np.inf
    acq[st.uniform(n) < 0.02] = np.nan
    mask = (st.uniform(n) < 0.75).astype(np.uint8)
    return torch.from_numpy(acq).cuda(), torch.from_numpy(mask).cuda()


def _outputs(q):
    return (torch.full((q,), -7, dtype=torch.int64, device="cuda"),
            torch.full((q,), 7.0, device="cuda"),
            torch.full((1,), -7, dtype=torch.int32, device="cuda"))


def test_static_topq_matches_workspace_topq_on_consecutive_calls(S):
    ctx = S.Context(torch.cuda.current_device())
    try:
        # large then small: the second call must not see the first call's partials
        for seed, n, q, use_mask in [(1, 1 << 21, 64, True), (2, 3001, 4, False), (3, 1 << 18, 16, True),
                                     (4, 17, 1, True)]:
            acq, mask = _case(seed, n)
            m = mask if use_mask else None
            want = _outputs(q)
            got = _outputs(q)
            S.scoot_select_topq(ctx, acq, n, q, *want, mask=m)
            S.scoot_select_topq_static(acq, n, q, *got, mask=m)
            torch.cuda.synchronize()
            for w, g in zip(want, got):
                assert torch.equal(w.cpu(), g.cpu()), (seed, n, q)
            assert int(got[2].item()) > 0
            # and the oracle's selection (Section 4.7 order) on the same values
            a_h = acq.cpu().numpy().astype(np.float64)
            oi, ov, oc = O.select_topq(a_h, None if m is None else mask.cpu().numpy(), q)
            assert int(got[2].item()) == oc
            assert got[0].cpu().numpy()[:oc].tolist() == oi.tolist()
            assert np.array_equal(got[1].cpu().numpy()[:oc].astype(np.float64), ov)
    finally:
        ctx.close()


def test_static_topq_rejects_sizes_beyond_its_limits(S):
    acq, mask = _case(5, 100)
    with pytest.raises(S.ScootError) as e:
        S.scoot_select_topq_static(acq, 100, 65, *_outputs(65))
    assert e.value.status == -6
    with pytest.raises(S.ScootError) as e:
        S.scoot_select_topq_static(acq, 1 << 32, 4, *_outputs(4))
    assert e.value.status == -6
