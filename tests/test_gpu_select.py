"""Token-level reduction (Sec. 3.1) on the GPU vs the oracle.

rolesub_select_tokens through the C ABI: kept indices are integers and the
gathered rows a copy, so both are compared bit for bit.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_18410_gb300 import build
    build.build()


def _check(oracle, scores, x, ratio):
    from paper_2608_18410_gb300 import rolesub
    keep, xk = rolesub.rolesub_select_tokens(torch.from_numpy(scores).cuda(), x, ratio)
    torch.cuda.synchronize()
    xh = x.cpu()
    xn = xh.view(torch.int16).numpy() if xh.dtype == torch.bfloat16 else xh.numpy()
    want_k, want_x = oracle.select_tokens(scores, xn, ratio)
    got_x = xk.cpu()
    got_x = got_x.view(torch.int16).numpy() if got_x.dtype == torch.bfloat16 else got_x.numpy()
    assert np.array_equal(keep.cpu().numpy(), want_k)
    assert np.array_equal(got_x, want_x)


@pytest.mark.parametrize("ratio", [0.015625, 0.03125, 0.0625])
def test_select_openvla_visual_budgets(oracle, ratio):
    # 64 episodes x 2 camera views x 256 tokens, hidden 4096, bf16
    rng = np.random.default_rng(60)
    scores = rng.standard_normal((64, 2, 256)).astype(np.float32)
    x = torch.randn(64, 2, 256, 4096, device="cuda").to(torch.bfloat16)
    _check(oracle, scores, x, ratio)


def test_select_ragged_ties_nan_and_float32(oracle):
    rng = np.random.default_rng(61)
    scores = rng.standard_normal((3, 2, 300)).astype(np.float32)
    scores[0, 0, :50] = 0.25                 # a block of exact ties
    scores[1, 1, 7] = np.nan
    scores[2, 0, :] = np.float32(1.0)        # every score equal
    x = torch.randn(3, 2, 300, 8, device="cuda")
    for r in (0.0625, 0.5, 1.0):
        _check(oracle, scores, x, r)
