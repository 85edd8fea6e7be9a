"""rolesub_compress_static: the compress call for callers that cannot
allocate device memory (a serving engine or control loop that reserves its
memory at start-up and forbids later allocation, or a plug-in whose host
gives it no scratch buffer). Its scratch is a fixed array inside the
library, so it takes no workspace.

The test goes through the C ABI: the allocation-free call must give what
rolesub_compress gives (same tolerance as the parity tests), on two calls
in a row (the array keeps the previous call's contents), must leave a clean
status word readable through rolesub_static_device_status, and must reject
a problem whose scratch does not fit. This file is collected last so that a
run stopping at the first failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest

from paper_2608_18410_gb300 import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

TOL = {"bf16": 1e-2, "f32": 1e-5}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_18410_gb300 import build
    build.build()


def _dev(x):
    if x.dtype == np.uint16:
        return torch.from_numpy(x.view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def _rows_close(a, b, wl, plan, tol):
    """Per (segment, head, token): max |a - b| <= tol * ||b's kept values||."""
    a = a.float().cpu().numpy()
    b = b.float().cpu().numpy()
    ds = wl.dh // wl.G
    for layer in range(wl.L):
        for sg in plan.segments:
            n, k = sg.n_tokens, sg.k
            if n == 0 or k == 0:
                continue
            sl = slice(sg.packed_off, sg.packed_off + wl.H * n * k * ds)
            x = a[layer, sl].reshape(wl.H, n, k * ds)
            y = b[layer, sl].reshape(wl.H, n, k * ds)
            nrm = np.linalg.norm(y, axis=2)
            err = np.abs(x - y).max(axis=2)
            assert np.all(err <= tol * nrm), float((err / np.maximum(nrm, 1e-30)).max())


@pytest.mark.parametrize("make", [synth.c0, synth.c1, lambda: synth.c2(64, 2).with_layers(4)])
def test_static_scratch_compress_matches_workspace_compress(make):
    from paper_2608_18410_gb300 import rolesub
    wl = make()
    inp = synth.gen_inputs(wl)
    rs = rolesub.RoleSub(wl.L, wl.H, wl.dh, wl.G, wl.C, wl.F, wl.dtype, wl.n_tok_array(), wl.k_array(),
                         wl.n_query_array())
    assert rs.ws_bytes <= rolesub.rolesub_static_scratch_bytes()
    d = {k: _dev(v) for k, v in inp.items()}
    args = (d["h"], d["v"], d["R"], d["W_re"], d["b_re"], d["W1"], d["b1"], d["W2"], d["b2"],
            wl.alpha_role, wl.alpha_lang)
    ref_p, ref_i = rs.compress(*args)
    torch.cuda.synchronize()
    for call in range(2):
        p, i = rs.new_outputs()
        p.fill_(float("nan"))
        i.fill_(255)
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        rolesub.rolesub_compress_static(rs.shape, rs.plan, rs.plan_dev, *args, p, i)
        torch.cuda.synchronize()
        if call == 1:
            assert torch.cuda.mem_get_info()[0] == free0, "the call must not allocate"
        assert rolesub.rolesub_static_device_status() == (0, 0), f"call {call}: device status"
        nidx = rs.plan.hdr.idx_bytes_per_layer
        assert torch.equal(i[:, :nidx], ref_i[:, :nidx]), f"call {call}: group indices differ"
        _rows_close(p, ref_p, wl, rs.plan, TOL[wl.dtype])


def test_static_scratch_rejects_problems_that_do_not_fit():
    from paper_2608_18410_gb300 import rolesub
    wl = synth.c4()
    shape = rolesub.make_shape(wl.L, wl.H, wl.dh, wl.G, wl.C, wl.F, wl.dtype)
    plan = rolesub.Plan(shape, wl.n_tok_array(), wl.k_array(), wl.n_query_array())
    assert plan.workspace_size() > rolesub.rolesub_static_scratch_bytes()
    fake = 1 << 20            # never touched: the size check comes first
    rc = rolesub.lib().rolesub_compress_static(ctypes.byref(shape), plan.host_ptr, fake, *([fake] * 9),
                                               0.1, 0.1, fake, fake, None)
    assert rc == 6            # ROLESUB_ETOOLARGE
    assert rolesub.rolesub_status_string(rc).startswith("problem needs more scratch")
