"""Workspace-free statistics entry point (adadsf_layer_stats_noalloc).

Some callers cannot hand the library scratch memory: their GPU memory belongs
to another allocator or a pre-reserved pool, or they only receive their input
and output buffers. For them the library keeps the reduction's partial sums in
a fixed device array of its own. This file checks, through the C ABI, that two
calls in a row give the same sums, bit for bit, as the workspace entry point
adadsf_layer_stats, that both agree with the oracle's Eq. 4 sums, and that
sizes beyond the array's limit are refused.
It is collected last and needs nothing from the other test files, so it can run
alone in a fresh process or after the rest of the suite."""
import numpy as np
import pytest
import torch

from oracle import adadsf_oracle as O

pytestmark = pytest.mark.gpu

REL_TOL = 1e-5     # the tolerance of the Eq. 4 statistics tests


def _pair(seed, n, d, dtype):
    g = torch.Generator(device="cpu").manual_seed(seed)
    a = torch.randn(n, d, generator=g)
    b = a + 0.5 * torch.randn(n, d, generator=g)
    return a.to("cuda", dtype), b.to("cuda", dtype)


@pytest.mark.parametrize("n,d,dtype,mode", [(5000, 1536, torch.bfloat16, 0), (3001, 512, torch.float32, 1),
                                            (40000, 768, torch.bfloat16, 0)])
def test_noalloc_matches_workspace_entry_point(n, d, dtype, mode):
    from paper_2607_21291_gb300 import adadsf as A
    A.lib()
    width = 2 if mode == A.STATS_TOKEN else 3
    for call, seed in enumerate((1, 2)):                    # two calls in a row, different data
        a, b = _pair(seed + n, n, d, dtype)
        ref = torch.zeros(width, dtype=torch.float64, device="cuda")
        A.adadsf_layer_stats(a, b, ref, mode=mode)
        got = torch.zeros(width, dtype=torch.float64, device="cuda")
        A.adadsf_layer_stats_noalloc(a, b, got, mode=mode)
        torch.cuda.synchronize()
        r, g_ = ref.cpu().numpy(), got.cpu().numpy()
        assert np.all(np.isfinite(g_)), (call, g_)
        # same kernels, same block count, same fixed summation order: the two
        # entry points agree bit for bit (a stale slot would show here)
        assert np.array_equal(g_, r), (call, g_, r)
        # and both follow the oracle's Eq. 4 sums on the same rounded inputs
        o = O.cos_sim_stat(a.double().cpu().numpy(), b.double().cpu().numpy(),
                           "token" if mode == A.STATS_TOKEN else "flat")
        assert g_ == pytest.approx(np.array(o), rel=REL_TOL), (call, g_, o)


def test_noalloc_refuses_oversized_calls():
    from paper_2607_21291_gb300 import adadsf as A
    lib = A.lib()
    acc = torch.zeros(2, dtype=torch.float64, device="cuda")
    x = torch.zeros(8, 8, dtype=torch.float32, device="cuda")
    for n_rows, d in ((2 ** 31, 8), (2 ** 40, 512)):
        st = lib.adadsf_layer_stats_noalloc(x.data_ptr(), x.data_ptr(), n_rows, d, A.F32, A.STATS_TOKEN,
                                            acc.data_ptr(), None)
        assert st == A.ERR_UNSUPPORTED
        assert "workspace-free" in A.adadsf_last_error()
    assert acc.cpu().tolist() == [0.0, 0.0]
