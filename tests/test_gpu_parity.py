"""CUDA path vs the fp64 oracle on the five workloads and on edge cases.

Every call goes through the C ABI (librolesub.so via the ctypes binding).
Full-size workloads are checked on sampled (layer, episode) pairs that the
oracle computes one by one, with the GPU running the whole launch.
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


def _run(wl, pairs):
    import parity
    inp = synth.gen_inputs(wl)
    gpu = parity.run_gpu(wl, inp)
    assert gpu["status"] == (0, 0)
    stats = [parity.check_layer_episode(wl, inp, gpu, l, e) for (l, e) in pairs]
    return gpu, stats


def test_c0_tiny_f32_full():
    wl = synth.c0()
    _, st = _run(wl, [(0, 0)])
    assert st[0]["exact_idx"] + st[0]["margin_idx"] == 64 + 16


def test_c1_one_layer_bf16_full():
    wl = synth.c1()
    _, st = _run(wl, [(0, 0)])
    assert st[0]["exact_idx"] + st[0]["margin_idx"] == 128


@pytest.mark.parametrize("nv,kv", synth.C2_POINTS)
def test_c2_stack_sampled_layers(nv, kv):
    wl = synth.c2(nv, kv)
    _run(wl, [(0, 0), (31, 0)])


def test_c3_near_ties_sampled_layers():
    import parity
    wl = synth.c3()
    inp = synth.gen_inputs(wl)
    gpu = parity.run_gpu(wl, inp)
    tot_margin = 0
    for l in (0, 9, 31):
        st = parity.check_layer_episode(wl, inp, gpu, l, 0)
        tot_margin += st["margin_idx"]
    assert tot_margin > 0, "the near-tie workload must exercise the margin rule"
    # exact ties (identical router rows and biases) resolve to the lower group
    # index on the GPU too: cluster 0 = groups 0..3 share score
    G = wl.G
    for l in (0, 31):
        k = wl.episodes[0].k_vis
        idx = gpu["idx"][l][:wl.episodes[0].n_vis * k].reshape(-1, k)
        for row in idx:
            sel = set(int(x) for x in row)
            in_c0 = sorted(g for g in sel if g < 4)
            assert in_c0 == list(range(len(in_c0))), row


@pytest.mark.slow
def test_c4_batched_ragged_full_size_sampled():
    wl = synth.c4()
    sizes = [ep.n_cache for ep in wl.episodes]
    e_big, e_small = int(np.argmax(sizes)), int(np.argmin(sizes))
    _run(wl, [(0, e_big), (31, e_small), (17, 5), (5, 40)])


# ---------------------------------------------------------------------------
# edge cases
# ---------------------------------------------------------------------------

def _wl(dtype, episodes, L=2, H=4, dh=None, G=None, C=8, F=32, seed=11):
    dh = dh or (128 if dtype == "bf16" else 64)
    G = G or (16 if dtype == "bf16" else 8)
    return synth.Workload(f"edge_{dtype}", dtype, L=L, H=H, dh=dh, G=G, C=C, F=F,
                          episodes=tuple(episodes), seed=seed)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_ragged_and_degenerate_segments(dtype):
    G = 16 if dtype == "bf16" else 8
    E = synth.Episode
    eps = [E(129, 7, 3, 3, G), E(1, 0, 1, 1, 2), E(0, 5, 2, 1, 1), E(0, 0, 4, 2, 2),
           E(65, 63, 64, 0, G), E(2, 3, 5, G, 0), E(40, 9, 9, G - 1, 1, n_prop=3, n_act=8)]
    wl = _wl(dtype, eps)
    _run(wl, [(l, e) for l in range(wl.L) for e in range(len(eps))])


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_long_cache_many_chunks(dtype):
    G = 16 if dtype == "bf16" else 8
    wl = _wl(dtype, [synth.Episode(400, 64, 64, 2, G // 2), synth.Episode(300, 20, 17, 4, 1)], L=1)
    _run(wl, [(0, 0), (0, 1)])


def test_attend_standalone_random_indices():
    import parity
    wl = synth.c4(num_episodes=6).with_layers(2)
    inp = synth.gen_inputs(wl)
    rs = parity.make_rolesub(wl)
    parity.check_attend_standalone(wl, inp, rs)


def test_attend_reads_keys_in_place_with_strides():
    """K inside a larger interleaved [rows][2][H][dh] KV buffer."""
    import parity
    wl = synth.c1()
    inp = synth.gen_inputs(wl)
    gpu = parity.run_gpu(wl, inp)
    rs = gpu["rs"]
    d = wl.d
    kv = np.zeros((wl.L, wl.rows, 2, d), np.uint16)
    kv[:, :, 0] = inp["K"]
    kv_t = parity.to_torch(kv, wl.dtype)
    packed = parity.to_torch(gpu["packed"], wl.dtype)
    idx = parity.to_torch(gpu["idx"], wl.dtype)
    o = rs.attend(parity.to_torch(inp["q"], wl.dtype), kv_t, packed, idx,
                  parity.to_torch(inp["R"], wl.dtype),
                  k_strides=(wl.rows * 2 * d, 2 * d, wl.dh))
    torch.cuda.synchronize()
    assert np.array_equal(parity.from_torch(o, wl.dtype), gpu["o"])


def test_bad_stored_index_is_reported_not_trapped():
    import parity
    wl = synth.c0()
    inp = synth.gen_inputs(wl)
    gpu = parity.run_gpu(wl, inp)
    rs = gpu["rs"]
    idx = gpu["idx"].copy()
    idx[0, 5] = 200                        # planted: group id >= S
    o = rs.attend(parity.to_torch(inp["q"], wl.dtype), parity.to_torch(inp["K"], wl.dtype),
                  parity.to_torch(gpu["packed"], wl.dtype), parity.to_torch(idx, wl.dtype),
                  parity.to_torch(inp["R"], wl.dtype))
    code, detail = rs.device_status()
    assert code == 4 and detail == 1       # ROLESUB_EDEVICE, cache row 1 (5 // k)
    assert np.all(np.isfinite(parity.from_torch(o, wl.dtype)))
    from paper_2608_18410_gb300 import rolesub
    rolesub.rolesub_reset_device_status(rs.workspace)
    assert rs.device_status() == (0, 0)


def test_bad_stored_index_bf16_tensor_core_path():
    import parity
    wl = synth.c1()
    inp = synth.gen_inputs(wl)
    gpu = parity.run_gpu(wl, inp)
    rs = gpu["rs"]
    idx = gpu["idx"].copy()
    idx[0, 4 * 7 + 2] = 99                 # vis token 7 (k = 4): group id >= S
    o = rs.attend(parity.to_torch(inp["q"], wl.dtype), parity.to_torch(inp["K"], wl.dtype),
                  parity.to_torch(gpu["packed"], wl.dtype), parity.to_torch(idx, wl.dtype),
                  parity.to_torch(inp["R"], wl.dtype))
    code, detail = rs.device_status()
    assert code == 4 and detail == 7
    assert np.all(np.isfinite(synth.widen(parity.from_torch(o, wl.dtype), wl.dtype)))
    from paper_2608_18410_gb300 import rolesub
    rolesub.rolesub_reset_device_status(rs.workspace)


def test_many_small_episodes_bf16():
    """More episodes than one attention launch covers (episode table limit)."""
    rng = np.random.default_rng(5)
    eps = [synth.Episode(int(rng.integers(0, 5)), int(rng.integers(0, 3)), int(rng.integers(0, 3)),
                         int(rng.choice([1, 2, 16])), int(rng.choice([0, 4, 16]))) for _ in range(600)]
    wl = _wl("bf16", eps, L=1, H=2, C=64, F=256)
    _run(wl, [(0, e) for e in (0, 1, 255, 511, 512, 513, 599)])


def test_repeated_calls_are_deterministic():
    import parity
    wl = synth.c1()
    inp = synth.gen_inputs(wl)
    a = parity.run_gpu(wl, inp)
    b = parity.run_gpu(wl, inp, rs=a["rs"])
    for key in ("packed", "idx", "o"):
        assert np.array_equal(a[key], b[key]), key


@pytest.mark.parametrize("H", [1, 3, 5])
def test_tensor_core_router_short_hidden(H):
    """The tensor-core router (F = 256, C = 64, S = 16) with d = 128, 384 and
    640: main loops of 2, 6 and 10 blocks, so the ring wraps a different
    number of times before the epilogue weights go into stage 0."""
    E = synth.Episode
    wl = synth.Workload(f"tc_router_h{H}", "bf16", L=2, H=H, dh=128, G=16, C=64, F=256,
                        episodes=(E(140, 20, 64, 3, 6), E(9, 40, 5, 8, 16)), seed=14)
    _run(wl, [(l, e) for l in range(2) for e in range(2)])


@pytest.mark.parametrize("extra", [-1, 1])
def test_persistent_kernels_uneven_item_counts(extra):
    """One 128-row router tile per layer, L = (SM count) - 1 or + 1. The
    persistent router launches min(items, SMs) CTAs, so with one item fewer
    than SMs every CTA takes exactly one item (the grid shrinks; no CTA is
    idle), and with one more one CTA takes a second item (a second trip round
    the ring, TMEM and barrier phases); the rotation's (head, layer, tile
    range) items wrap unevenly over its CTAs."""
    L = torch.cuda.get_device_properties(0).multi_processor_count + extra
    E = synth.Episode
    wl = synth.Workload(f"persist_l{L}", "bf16", L=L, H=2, dh=128, G=16, C=64, F=256,
                        episodes=(E(128, 8, 16, 4, 16),), seed=16)
    _run(wl, [(0, 0), (L // 2, 0), (L - 2, 0), (L - 1, 0)])


def test_attention_split_over_launches():
    """More units than one launch holds (512 per CTA): 320 tiny episodes x 32
    heads x 8 layers = 81,920 units, so the call runs two launches; sampled
    pairs sit in both."""
    E = synth.Episode
    eps = [E(8 + (i % 5), 4 + (i % 3), 1 + (i % 2), 2 + (i % 3), 4) for i in range(320)]
    wl = synth.Workload("many_units", "bf16", L=8, H=32, dh=128, G=16, C=8, F=32, episodes=tuple(eps), seed=15)
    _run(wl, [(0, 0), (0, 319), (3, 160), (7, 1), (7, 318)])
