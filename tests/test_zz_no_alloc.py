"""bfasgd_select_compact_noalloc: the send decision and compaction for
callers that may not allocate device memory (a framework that owns every
allocation through its own pool, a fixed device-memory budget, or a loop
that cannot take the implicit synchronisation of cudaMalloc).  It must give
exactly what the handle-based bfasgd_select_compact gives, call after call,
and it must not allocate.  Collected last so that a failure here stops a
-x run only after every other test has run."""

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

SEED = 0x5EED_0F_B_FA5
EPS_B = 1e-8


def _f():
    from paper_1601_04033_gb300 import fasgd
    return fasgd


def _outputs(P, device):
    import torch
    return (torch.full((P,), -1, dtype=torch.int32, device=device),
            torch.full((P,), float("nan"), dtype=torch.float32, device=device),
            torch.full((1,), -1, dtype=torch.int64, device=device))


@pytest.mark.parametrize("P", [1_000_003, 1 << 24])
def test_noalloc_matches_handle_two_calls_in_a_row(P):
    import torch
    f = _f()
    rng = np.random.default_rng(P)
    g = torch.from_numpy((rng.standard_normal(P) * 0.1).astype(np.float32)).cuda()
    v = torch.from_numpy((10 ** rng.uniform(0, 2, P)).astype(np.float32)).cuda()
    c = 40.0
    srv = f.Server(P, 4, 0.001, f.FASGD, c_push=c, eps_b=EPS_B, seed=SEED)
    stream = torch.cuda.current_stream()
    client = 2
    for push_no in range(2):            # two calls in a row, same client
        hi, hv, hn = _outputs(P, "cuda")
        srv.select_compact(client, g, hi, hv, hn, v=v)
        ni, nv, nn = _outputs(P, "cuda")
        rc = f.bfasgd_select_compact_noalloc(P, g.data_ptr(), v.data_ptr(), c, EPS_B, SEED,
                                             client, push_no, ni.data_ptr(), nv.data_ptr(),
                                             nn.data_ptr(), stream.cuda_stream)
        assert rc == f.OK, f.fasgd_last_error(None)
        torch.cuda.synchronize()
        m = int(hn.item())
        assert int(nn.item()) == m and 0 < m < P
        assert torch.equal(ni[:m], hi[:m])
        assert torch.equal(nv[:m].view(torch.int32), hv[:m].view(torch.int32))
    srv.close()


def test_noalloc_allocates_nothing_and_rejects_oversize():
    import torch
    f = _f()
    P = 300_001
    g = torch.randn(P, device="cuda")
    v = torch.rand(P, device="cuda") * 10 + 1
    idx, val, n = _outputs(P, "cuda")
    stream = torch.cuda.current_stream().cuda_stream
    args = (g.data_ptr(), v.data_ptr(), 5.0, EPS_B, SEED, 0, 0, idx.data_ptr(), val.data_ptr(),
            n.data_ptr(), stream)
    assert f.bfasgd_select_compact_noalloc(P, *args) == f.OK      # first call: set-up
    torch.cuda.synchronize()
    free_before = torch.cuda.mem_get_info()[0]
    for _ in range(3):
        assert f.bfasgd_select_compact_noalloc(P, *args) == f.OK
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free_before
    big = f.NOALLOC_PMAX + 1
    assert f.bfasgd_select_compact_noalloc(big, *args) == f.EINVAL
    assert "static scratch" in f.fasgd_last_error(None)
    assert f.bfasgd_select_compact_noalloc(0, *args) == f.EINVAL


def test_noalloc_sizes_in_turn_match_oracle():
    """Calls of different sizes share the one scratch array: every call must
    see only its own tile status words, whatever an earlier, larger or
    smaller call left there."""
    import torch
    import oracle
    f = _f()
    stream = torch.cuda.current_stream().cuda_stream
    for k, P in enumerate([1 << 24, 5, 8193, (1 << 24) - 3, 100_000, 8192]):
        rng = np.random.default_rng(1000 + k)
        g = (rng.standard_normal(P) * 0.1).astype(np.float32)
        v = (10 ** rng.uniform(-1, 2, P)).astype(np.float32)
        c = np.float32(30.0)
        g_t, v_t = torch.from_numpy(g).cuda(), torch.from_numpy(v).cuda()
        idx, val, n = _outputs(P, "cuda")
        rc = f.bfasgd_select_compact_noalloc(P, g_t.data_ptr(), v_t.data_ptr(), float(c), EPS_B,
                                             SEED, 3, k, idx.data_ptr(), val.data_ptr(),
                                             n.data_ptr(), stream)
        assert rc == f.OK, f.fasgd_last_error(None)
        torch.cuda.synchronize()
        oi, ov = oracle.select(g, v, c, EPS_B, SEED, 3, k)
        m = int(n.item())
        assert m == oi.size, (P, m, oi.size)
        assert np.array_equal(idx[:m].cpu().numpy(), oi)
        assert np.array_equal(val[:m].cpu().numpy().view(np.int32), ov.view(np.int32))
