"""Failure handling on the device: a bounded wait that runs out.

Every tensor-core kernel waits on mbarriers through one bounded loop; when a
wait gives up it records ROLESUB_ETIMEOUT and its site in the status word and
raises the CTA's abort flag, so that the CTA's other waits return at once.
rolesub_wait_selftest runs that loop in a small kernel on an mbarrier that
nothing arrives on (no copy or tensor-core work in flight), with a limit of a
few milliseconds. The test checks the status word, that both waits came back
promptly, and that the context stays usable: a compress + attend call after it
is clean and bit-identical to the same call before it.
"""
import time

import numpy as np
import pytest

from paper_2608_18410_gb300 import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

ETIMEOUT = 5
SITE_LEADER = 900


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


def _step(rs, d, wl):
    p, i = rs.new_outputs()
    rs.compress(d["h"], d["v"], d["R"], d["W_re"], d["b_re"], d["W1"], d["b1"], d["W2"], d["b2"],
                wl.alpha_role, wl.alpha_lang, packed=p, idx=i)
    o = rs.attend(d["q"], d["K"], p, i, d["R"])
    torch.cuda.synchronize()
    return p.clone(), i.clone(), o.clone()


@pytest.mark.parametrize("limit_ms", [2, 20])
def test_wait_that_runs_out_reports_and_returns(limit_ms):
    from paper_2608_18410_gb300 import rolesub
    wl = synth.c1()
    inp = synth.gen_inputs(wl)
    rs = rolesub.RoleSub(wl.L, wl.H, wl.dh, wl.G, wl.C, wl.F, wl.dtype, wl.n_tok_array(), wl.k_array(),
                         wl.n_query_array())
    d = {k: _dev(v) for k, v in inp.items()}
    before = _step(rs, d, wl)
    assert rs.device_status() == (0, 0)

    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    out = torch.full((4,), -1, dtype=torch.int64, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    rolesub.rolesub_wait_selftest(limit_ms * 1_000_000, ws, out)
    code, site = rolesub.rolesub_get_device_status(ws)
    wall = time.perf_counter() - t0
    leader_ok, leader_ns, follower_ok, follower_ns = out.cpu().tolist()
    assert (code, site) == (ETIMEOUT, SITE_LEADER)
    assert leader_ok == 0 and follower_ok == 0
    assert leader_ns >= limit_ms * 1_000_000, leader_ns
    assert leader_ns < limit_ms * 1_000_000 + 50_000_000, leader_ns
    # the follower had a two-second limit and came back through the abort flag
    assert follower_ns < limit_ms * 1_000_000 + 50_000_000, follower_ns
    assert wall < 1.0, wall

    # the context is still usable and the library's own calls are unaffected
    after = _step(rs, d, wl)
    assert rs.device_status() == (0, 0)
    for x, y in zip(before, after):
        assert torch.equal(x.view(torch.uint8) if x.dtype != torch.uint8 else x,
                           y.view(torch.uint8) if y.dtype != torch.uint8 else y)
