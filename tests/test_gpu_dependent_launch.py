"""A call reads nothing that its workspace held before the call.

Within a call, every kernel after the first is started as a programmatic
dependent of the one before it, so it is resident while its predecessor
still writes. The language context, the per-episode router terms, the budget
scores and the store records are written and read inside the call. With few
layers the first kernel's grid is small and its dependents start at once,
and a read of those buffers that is not ordered after the dependent's wait
sees the workspace's old contents. (Such a read was found: the language-bias
kernels read the context through the read-only path, ahead of the wait, and
routed differently at 1-8 layers than at 32.)

Each case fills the whole workspace with 0xFF bytes (NaN as fp32), clears the
status word through rolesub_reset_device_status, and calls again: packed
values, indices, counts and outputs must equal those of the first call on a
zeroed workspace bit for bit, for 1 and 4 layers, both language-bias forms
(64 episodes: the tensor-core bias; 2 episodes: the matrix-vector one), the
additive router and the per-token budget pair.
"""
import dataclasses

import numpy as np
import pytest

from paper_2608_18410_gb300 import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_18410_gb300 import build
    build.build()


def _poison(rs):
    from paper_2608_18410_gb300 import rolesub
    rs.workspace.fill_(0xFF)
    rolesub.rolesub_reset_device_status(rs.workspace)


def _workload(L, E):
    wl = synth.c4(num_episodes=E).with_layers(L)
    return dataclasses.replace(wl, seed=wl.seed + 100 * L + E)


@pytest.mark.parametrize("L,E", [(1, 64), (4, 64), (1, 2)])
def test_fixed_router_ignores_old_workspace(L, E):
    import parity
    wl = _workload(L, E)
    inp = synth.gen_inputs(wl)
    rs = parity.make_rolesub(wl)
    dev = {k: parity.to_torch(v, wl.dtype) for k, v in inp.items()}

    def call():
        packed, idx = rs.compress(dev["h"], dev["v"], dev["R"], dev["W_re"], dev["b_re"], dev["W1"], dev["b1"],
                                  dev["W2"], dev["b2"], wl.alpha_role, wl.alpha_lang)
        o = rs.attend(dev["q"], dev["K"], packed, idx, dev["R"])
        torch.cuda.synchronize()
        assert rs.device_status() == (0, 0)
        return packed.clone(), idx.clone(), o.clone()

    ref = call()
    for _ in range(3):
        _poison(rs)
        got = call()
        for a, b in zip(ref, got):
            assert torch.equal(a, b)


@pytest.mark.parametrize("L", [1, 4])
def test_additive_and_budget_ignore_old_workspace(L):
    import parity
    wl = dataclasses.replace(_workload(L, 64), C=6)
    inp = synth.gen_inputs(wl)
    add = synth.gen_additive_weights(wl)
    u = torch.from_numpy(np.ascontiguousarray(synth.gen_priority(wl), np.float32)).cuda()
    rs = parity.make_rolesub(wl)
    dev = {k: parity.to_torch(v, wl.dtype) for k, v in inp.items()}
    da = {k: parity.to_torch(v, wl.dtype) for k, v in add.items()}

    def call():
        packed, idx = rs.compress_additive(dev["h"], dev["v"], dev["R"], dev["W_re"], dev["b_re"], da["W_v"],
                                           da["b_v"], da["W_role"], da["W_l"], da["b_l"], wl.alpha_role,
                                           wl.alpha_lang)
        o = rs.attend(dev["q"], dev["K"], packed, idx, dev["R"])
        bp, bi, kt = rs.compress_budget(dev["h"], dev["v"], dev["R"], dev["W_re"], dev["b_re"], da["W_v"],
                                        da["b_v"], da["W_role"], da["W_l"], da["b_l"], u, wl.alpha_role,
                                        wl.alpha_lang)
        bo = rs.attend_budget(dev["q"], dev["K"], bp, bi, kt, dev["R"])
        torch.cuda.synchronize()
        assert rs.device_status() == (0, 0)
        return [t.clone() for t in (packed, idx, o, bp, bi, kt, bo)]

    ref = call()
    for _ in range(3):
        _poison(rs)
        got = call()
        for a, b in zip(ref, got):
            assert torch.equal(a, b)
