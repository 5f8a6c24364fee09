"""slorr_frob_sq_noalloc: the squared Frobenius norm computed with no device
allocation, for callers that cannot hand the library a workspace (code running
under stream capture, or under a framework that owns all device memory).

Checked through the C ABI against the workspace-based path (the norm pass of
slorr_run_steps, read back from the workspace) on two calls in a row: a large
matrix first, then a smaller ragged one, so that partial sums the first call
left in the shared fixed scratch would show up if the second call read them.
This file is collected last on purpose.
"""

import numpy as np
import pytest

import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-5   # the fp32 tolerance of the parity tests


def _workspace_frob_sq(W, dtype="f32"):
    from paper_2607_08754_gb300.slorr import Regularizer
    reg = Regularizer([W.shape], compute="fp32", dtype=dtype)
    w = torch.from_numpy(W).cuda()
    if dtype == "bf16":
        w = w.to(torch.bfloat16)
    reg.run_steps([w], 0)
    torch.cuda.synchronize()
    return reg.scalars(0)[0]


def test_noalloc_frob_sq_matches_workspace_path_on_two_calls():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    mats = [workloads.random_matrix((1024, 4096), seed=5001, std=0.02),
            workloads.random_matrix((320, 147), seed=5002, std=0.3)]
    refs = [_workspace_frob_sq(W) for W in mats]
    stream = torch.cuda.current_stream().cuda_stream
    outs = []
    for W in mats:                                   # two calls in a row
        w = torch.from_numpy(W).cuda()
        out = torch.full((1,), float("nan"), dtype=torch.float64, device="cuda")
        slorr.slorr_frob_sq_noalloc(w.data_ptr(), W.shape[0], W.shape[1], 0, out.data_ptr(), stream)
        torch.cuda.synchronize()
        outs.append(out.item())
    for got, ref, W in zip(outs, refs, mats):
        exact = float(np.sum(W.astype(np.float64) ** 2))
        assert got == pytest.approx(ref, rel=TOL)
        assert got == pytest.approx(exact, rel=TOL)


def test_noalloc_frob_sq_bf16_on_two_calls():
    """bf16 weights (dtype SLORR_BF16): two calls in a row against the
    workspace path with bf16 storage and an fp64 sum of the bf16 values."""
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    mats = [workloads.random_matrix((2048, 1536), seed=5003, std=0.02),
            workloads.random_matrix((77, 300), seed=5004, std=0.5)]
    refs = [_workspace_frob_sq(W, "bf16") for W in mats]
    stream = torch.cuda.current_stream().cuda_stream
    for W, ref in zip(mats, refs):
        w = torch.from_numpy(W).cuda().to(torch.bfloat16)
        out = torch.full((1,), float("nan"), dtype=torch.float64, device="cuda")
        slorr.slorr_frob_sq_noalloc(w.data_ptr(), W.shape[0], W.shape[1], 1, out.data_ptr(), stream)
        torch.cuda.synchronize()
        exact = float(torch.sum(w.double() ** 2).item())
        assert out.item() == pytest.approx(ref, rel=TOL)
        assert out.item() == pytest.approx(exact, rel=TOL)


def test_noalloc_rejects_oversized_matrix():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    w = torch.zeros(4, device="cuda")
    out = torch.zeros(1, dtype=torch.float64, device="cuda")
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_frob_sq_noalloc(w.data_ptr(), 65536, 65536, 0, out.data_ptr(), 0)
    assert e.value.status == 1 and "too large" in str(e.value)
