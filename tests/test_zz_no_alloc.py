"""jet_score_candidates_noalloc: scoring for callers that cannot allocate.

Some callers of this library cannot call cudaMalloc - a host application that
owns all device memory and hands a plug-in only its tensors, or a serving loop
that must not allocate (cudaMalloc can synchronise the device and can fail
under memory pressure) while it runs. For them the library offers one entry
point that uses a fixed scratch array inside the library instead of a
caller-provided workspace. This file checks it through the C ABI against the
workspace entry point, twice in a row (the array is shared by every call and
keeps the previous call's contents). It is named to be collected last.
"""
import numpy as np
import pytest

import jet_synth
from gpu_common import TOL_LOGPROB, build_step

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["tiny", "dense27b_mc", "binary"])
def test_noalloc_matches_workspace_entry_point(jet, name):
    import torch
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required for -m gpu tests")
    p = jet_synth.make_problem(name)
    step, x, w_lm = build_step(jet, p)
    lay, dims = step.layout, step.dims
    jet.jet_score_candidates(lay, dims, x["hidden"], w_lm, step.tok_logprob, step.cand_score,
                             step.ws)
    torch.cuda.synchronize()
    ref_ell = step.tok_logprob.cpu().numpy()
    ref_s = step.cand_score.cpu().numpy()
    for _ in range(2):
        ell = torch.full_like(step.tok_logprob, float("nan"))
        s = torch.full_like(step.cand_score, float("nan"))
        jet.jet_score_candidates_noalloc(lay, dims, x["hidden"], w_lm, ell, s)
        torch.cuda.synchronize()
        assert jet.jet_device_status() == 0
        np.testing.assert_allclose(ell.cpu().numpy(), ref_ell, rtol=0, atol=TOL_LOGPROB)
        np.testing.assert_allclose(s.cpu().numpy(), ref_s, rtol=0, atol=TOL_LOGPROB)


def test_noalloc_rejects_batches_beyond_its_scratch(jet):
    # 2,000 rows over a 151,936-entry vocabulary need about 19 MB of scratch,
    # more than the fixed 16 MiB: the call must refuse before launching
    V = 151936
    hl = jet.jet_layout_build([4], [1], [2001], list(range(2001)), V)
    dims = jet.make_dims(jet.DTYPE_BF16, D=64)
    with pytest.raises(jet.JetError) as e:
        jet.jet_score_candidates_noalloc(hl, dims, 1 << 40, 1 << 40, 1 << 40, 1 << 40, stream=0)
    assert e.value.status == 6  # JET_ERR_CAPACITY
