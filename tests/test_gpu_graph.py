"""compress + attend captured in a CUDA graph and replayed.

The calls enqueue only kernel launches on the caller's stream (tensor maps
are encoded and launch attributes set on the host), so a captured step
replays bit-identically to an eager one.
"""
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


@pytest.mark.parametrize("make", [synth.c1, lambda: synth.c4(num_episodes=8).with_layers(2)])
def test_graph_replay_matches_eager(make):
    import parity
    wl = make()
    inp = synth.gen_inputs(wl)
    rs = parity.make_rolesub(wl)
    d = {k: parity.to_torch(v, wl.dtype) for k, v in inp.items()}
    packed, idx = rs.new_outputs()
    o = torch.empty((wl.L, max(wl.q_rows, 1), wl.d), dtype=rs.tdtype, device="cuda")

    def step():
        rs.compress(d["h"], d["v"], d["R"], d["W_re"], d["b_re"], d["W1"], d["b1"], d["W2"], d["b2"],
                    wl.alpha_role, wl.alpha_lang, packed=packed, idx=idx)
        rs.attend(d["q"], d["K"], packed, idx, d["R"], o=o)

    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        step()                                   # eager, also warms the library up
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    ref_idx, ref_o = idx.clone(), o.clone()
    packed.zero_()
    idx.zero_()
    o.zero_()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(idx, ref_idx)
    assert torch.equal(o.view(torch.int16) if o.dtype == torch.bfloat16 else o,
                       ref_o.view(torch.int16) if ref_o.dtype == torch.bfloat16 else ref_o)
    assert rs.device_status() == (0, 0)
