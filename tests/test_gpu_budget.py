"""Per-token value budgets (Sec. 3.5) on the GPU vs the oracle.

rolesub_compress_budget (additive score, priority pi = u . a, the
allocator's counts, top-K_i at prefix offsets) and rolesub_attend_budget over
the cache it wrote, through the C ABI; the fp64 oracle routes with
route_layer_budget and packs / attends with the numpy budget restatement.
Counts must meet each segment's budget and follow every priority order wider
than 1e-4 (exact where a token's priority is that far from all others);
indices, packed values and outputs are then checked on the GPU's counts with
the margin and row-norm rules of the fixed-k tests.
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


def _run(wl, pairs):
    import parity
    inp = synth.gen_inputs(wl)
    add = synth.gen_additive_weights(wl)
    u = synth.gen_priority(wl)
    gpu = parity.run_gpu_budget(wl, inp, add, u)
    assert gpu["status"] == (0, 0)
    return gpu, [parity.check_budget_layer_episode(wl, inp, add, u, gpu, l, e) for (l, e) in pairs]


def test_budget_oft_layer():
    wl = dataclasses.replace(synth.c1(), C=6)
    _, st = _run(wl, [(0, 0)])
    assert st[0]["exact_k"] > 100 and st[0]["exact_idx"] > 100


@pytest.mark.parametrize("k_vis", [1, 4, 12, 15])
def test_budget_targets_including_saturation(k_vis):
    """k_vis = 12 and 15 make the best ranks saturate at S = 16."""
    E = synth.Episode
    wl = synth.Workload("budget_k", "bf16", L=2, H=4, dh=128, G=16, C=6, F=8,
                        episodes=(E(150, 20, 64, k_vis, 5), E(33, 9, 7, k_vis, 16)), seed=31)
    _run(wl, [(l, e) for l in range(2) for e in range(2)])


def test_budget_ragged_and_degenerate_segments():
    E = synth.Episode
    eps = [E(129, 7, 3, 3, 16), E(1, 0, 1, 1, 2), E(0, 5, 2, 1, 1), E(0, 0, 4, 2, 2),
           E(65, 63, 64, 0, 16), E(2, 3, 5, 16, 0), E(40, 9, 9, 15, 1, n_prop=3, n_act=8),
           E(300, 16, 64, 8, 8)]
    wl = synth.Workload("budget_edge", "bf16", L=2, H=4, dh=128, G=16, C=6, F=8, episodes=tuple(eps), seed=32)
    _run(wl, [(l, e) for l in range(wl.L) for e in range(len(eps))])


def test_budget_batched_ragged_episodes():
    wl = dataclasses.replace(synth.c4(num_episodes=12), C=6, L=2)
    _run(wl, [(l, e) for l in range(2) for e in (0, 4, 9, 11)])


@pytest.mark.slow
def test_budget_c4_full_size_sampled():
    wl = dataclasses.replace(synth.c4(), C=6)
    sizes = [ep.n_cache for ep in wl.episodes]
    e_big, e_small = int(np.argmax(sizes)), int(np.argmin(sizes))
    _run(wl, [(0, e_big), (31, e_small), (17, 5)])


def test_budget_attend_reports_corrupt_counts():
    """A count above S and counts that overrun a segment's budget are
    reported in the status word and stored nothing; nothing traps."""
    import parity
    E = synth.Episode
    wl = synth.Workload("budget_bad", "bf16", L=1, H=2, dh=128, G=16, C=6, F=8,
                        episodes=(E(20, 4, 8, 4, 4),), seed=33)
    inp = synth.gen_inputs(wl)
    add = synth.gen_additive_weights(wl)
    u = synth.gen_priority(wl)
    gpu = parity.run_gpu_budget(wl, inp, add, u)
    assert gpu["status"] == (0, 0)
    rs = gpu["rs"]
    dev = {k: parity.to_torch(v, wl.dtype) for k, v in inp.items()}
    packed = parity.to_torch(gpu["packed"], wl.dtype)
    idx = torch.from_numpy(gpu["idx"]).cuda()
    for bad in (17, 16):   # 17 > S; 16 on one row overruns the segment's 80 groups
        kt = gpu["ktok"].copy()
        kt[0, 3] = bad
        rs.attend_budget(dev["q"], dev["K"], packed, idx, torch.from_numpy(kt).cuda(), dev["R"])
        torch.cuda.synchronize()
        code, detail = rs.device_status()
        assert code == 4, (bad, code)
        from paper_2608_18410_gb300 import rolesub
        rolesub.rolesub_reset_device_status(rs.workspace)
        torch.cuda.synchronize()


def test_budget_rejects_unsupported_geometry():
    from paper_2608_18410_gb300 import rolesub as R
    import parity
    wl = synth.Workload("budget_f32", "f32", L=1, H=2, dh=64, G=8, C=6, F=8,
                        episodes=(synth.Episode(4, 2, 1, 2, 2),), seed=0)
    rs = parity.make_rolesub(wl)
    z = torch.zeros(1 << 16, device="cuda")
    with pytest.raises(R.RoleSubError) as ei:
        rs.compress_budget(z, z, z, z, z, z, z, z, z, z, z)
    assert ei.value.code == 2
