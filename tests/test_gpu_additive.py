"""Additive routing score (Sec. 3.4, Eq. routingscore) on the GPU vs the oracle.

rolesub_compress_additive through the C ABI, then rolesub_attend over the
cache it packed; the fp64 oracle routes with compress_layer_linear. Indices
are bit-exact where the oracle's top-k margin exceeds 1e-4 (else any valid
top-k), packed values and outputs within 1e-2 (bf16) / 1e-5 (fp32) of the
row norm. Shapes use the paper's C = 6 role components (Sec. 4.1) unless a
case widens C to reach more TMEM column chunks of the tensor-core epilogue.
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
    gpu = parity.run_gpu(wl, inp, add=add)
    assert gpu["status"] == (0, 0)
    stats = [parity.check_layer_episode(wl, inp, gpu, l, e, add=add) for (l, e) in pairs]
    return gpu, stats


def test_additive_c0_tiny_f32():
    wl = dataclasses.replace(synth.c0(), C=6)
    _, st = _run(wl, [(0, 0)])
    assert st[0]["exact_idx"] + st[0]["margin_idx"] == 64 + 16


def test_additive_c1_oft_layer_bf16_tensor_core():
    wl = dataclasses.replace(synth.c1(), C=6)
    _, st = _run(wl, [(0, 0)])
    assert st[0]["exact_idx"] + st[0]["margin_idx"] == 128
    assert st[0]["exact_idx"] > 100


@pytest.mark.parametrize("C", [1, 6, 40, 64, 240])
def test_additive_role_widths_bf16(C):
    """C spans one to eight 32-column TMEM chunks (S + C up to 256)."""
    E = synth.Episode
    wl = synth.Workload("add_C", "bf16", L=2, H=4, dh=128, G=16, C=C, F=8,
                        episodes=(E(150, 20, 5, 3, 5), E(7, 3, 2, 1, 15)), seed=21)
    _run(wl, [(l, e) for l in range(2) for e in range(2)])


@pytest.mark.parametrize("dtype,G", [("f32", 8), ("bf16", 8), ("bf16", 16)])
def test_additive_ragged_and_degenerate_segments(dtype, G):
    E = synth.Episode
    eps = [E(129, 7, 3, 3, G), E(1, 0, 1, 1, 2), E(0, 5, 2, 1, 1), E(0, 0, 4, 2, 2),
           E(65, 63, 64, 0, G), E(2, 3, 5, G, 0), E(40, 9, 9, G - 1, 1, n_prop=3, n_act=8)]
    dh = 128 if dtype == "bf16" else 64
    wl = synth.Workload(f"add_edge_{dtype}", dtype, L=2, H=4, dh=dh, G=G, C=6, F=8, episodes=tuple(eps),
                        seed=12)
    _run(wl, [(l, e) for l in range(wl.L) for e in range(len(eps))])


def test_additive_near_ties_use_margin_rule():
    wl = dataclasses.replace(synth.c3(), C=6, L=3)
    _, st = _run(wl, [(0, 0), (2, 0)])
    assert sum(s["margin_idx"] for s in st) > 0


def test_additive_batched_ragged_episodes():
    wl = dataclasses.replace(synth.c4(num_episodes=12), C=6, L=2)
    _run(wl, [(l, e) for l in range(2) for e in (0, 3, 7, 11)])


def test_additive_rejects_oversized_role_dim():
    from paper_2608_18410_gb300 import rolesub as R
    wl = synth.Workload("add_big_C", "f32", L=1, H=2, dh=8, G=4, C=5000, F=8,
                        episodes=(synth.Episode(4, 2, 1, 2, 2),), seed=0)
    rs = __import__("parity").make_rolesub(wl)
    z = torch.zeros(1 << 16, device="cuda")
    with pytest.raises(R.RoleSubError) as ei:
        rs.compress_additive(z, z, z, z, z, z, z, z, z, z)
    assert ei.value.code == 2


@pytest.mark.slow
def test_additive_c4_full_size_sampled():
    """The batched ragged workload at full size (64 episodes, 32 layers) in
    the launch configuration the benchmark times, checked on sampled
    (layer, episode) pairs."""
    wl = dataclasses.replace(synth.c4(), C=6)
    sizes = [ep.n_cache for ep in wl.episodes]
    e_big, e_small = int(np.argmax(sizes)), int(np.argmin(sizes))
    _run(wl, [(0, e_big), (31, e_small), (17, 5), (5, 40)])
