"""The dense-rotation geometry (one d x d R per layer, Sec. 4.1) on the GPU vs
the oracle.

rolesub_compress_dense / rolesub_attend_dense through the C ABI. Indices come
from the same router as the per-head path (bit-exact where the top-k margin
exceeds 1e-4); packed groups are compared with z = R^T v over all d dims on
the GPU's indices (1e-2 of the token's ||z||), outputs with the numpy dense
oracle on the GPU's packed cache (1e-2 of each (query, head) row norm).
"""
import numpy as np
import pytest

import oracle
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
    Rd = synth.gen_dense_rotation(wl)
    rs = parity.make_rolesub(wl)
    dev = {k: parity.to_torch(v, wl.dtype) for k, v in inp.items()}
    dR = parity.to_torch(Rd, wl.dtype)
    packed, idx = rs.compress_dense(dev["h"], dev["v"], dR, dev["W_re"], dev["b_re"], dev["W1"], dev["b1"],
                                    dev["W2"], dev["b2"], wl.alpha_role, wl.alpha_lang)
    o = rs.attend_dense(dev["q"], dev["K"], packed, idx, dR)
    torch.cuda.synchronize()
    assert rs.dense_device_status() == (0, 0)
    gp = synth.widen(parity.from_torch(packed, wl.dtype), wl.dtype)
    gi = idx.cpu().numpy()
    go = synth.widen(parity.from_torch(o, wl.dtype), wl.dtype)
    glob = oracle.layout(wl.n_tok_array(), wl.k_array(), wl.H, wl.dh, wl.G)
    G, H, dh, d = wl.G, wl.H, wl.dh, wl.d
    gw = d // G
    for (l, e) in pairs:
        ep = wl.episodes[e]
        n_tok = np.array(ep.n_tok(), np.int32)
        kk = np.array(ep.k(G), np.int32)
        spec = oracle.Spec(H, dh, G, wl.C, wl.F, n_tok[None], kk[None], [ep.n_query])
        loc = spec.lay
        r0 = int(glob["row_off"][4 * e])
        r1 = r0 + ep.n_cache
        q0 = int(sum(x.n_query for x in wl.episodes[:e]))
        W = lambda name: synth.widen(inp[name][l], wl.dtype)
        h = synth.widen(inp["h"][l, r0:r1], wl.dtype)
        v = synth.widen(inp["v"][l, r0:r1], wl.dtype)
        R = synth.widen(Rd[l], wl.dtype)
        ref = oracle.compress_layer(spec, h, v, W("R"), W("W_re"), inp["b_re"][l].astype(np.float64), W("W1"),
                                    inp["b1"][l].astype(np.float64), W("W2"), inp["b2"][l].astype(np.float64),
                                    wl.alpha_role, wl.alpha_lang, want_z=False)
        idx_loc = np.zeros(max(loc["idx_bytes"], 1), np.uint8)
        pk_loc = np.zeros(max(loc["packed_elems"], 1))
        for m in range(4):
            n, k = int(n_tok[m]), int(kk[m])
            if n == 0 or k == 0:
                continue
            gs = gi[l, glob["idx_off"][4 * e + m]: glob["idx_off"][4 * e + m] + n * k].reshape(n, k)
            os_ = ref["idx"][loc["idx_off"][m]: loc["idx_off"][m] + n * k].reshape(n, k)
            for i in range(n):
                if k == G or ref["margin"][int(loc["row_off"][m]) + i] > 1e-4:
                    assert np.array_equal(gs[i], os_[i]), (l, e, m, i)
            idx_loc[loc["idx_off"][m]: loc["idx_off"][m] + n * k] = gs.reshape(-1)
            pk_loc[loc["packed_off"][m]: loc["packed_off"][m] + n * k * gw] = \
                gp[l, glob["packed_off"][4 * e + m]: glob["packed_off"][4 * e + m] + n * k * gw]
        want = oracle.pack_layer_dense(spec, v, R, idx_loc)
        z = v @ R
        for m in range(4):
            n, k, rs_ = int(n_tok[m]), int(kk[m]), int(loc["row_off"][m])
            if n == 0 or k == 0:
                continue
            a = pk_loc[loc["packed_off"][m]: loc["packed_off"][m] + n * k * gw].reshape(n, k * gw)
            b = want[loc["packed_off"][m]: loc["packed_off"][m] + n * k * gw].reshape(n, k * gw)
            nrm = np.linalg.norm(z[rs_:rs_ + n], axis=1)
            assert np.all(np.abs(a - b).max(axis=1) <= 1e-2 * nrm), (l, e, m)
        if ep.n_query:
            qe = synth.widen(inp["q"][l, q0:q0 + ep.n_query], wl.dtype)
            Ke = synth.widen(inp["K"][l, r0:r1], wl.dtype)
            o_ref = oracle.attend_layer_dense(spec, qe, Ke, pk_loc, idx_loc, R).reshape(-1, H, dh)
            o_gpu = go[l, q0:q0 + ep.n_query].reshape(-1, H, dh)
            nrm = np.linalg.norm(o_ref, axis=2)
            err = np.abs(o_gpu - o_ref).max(axis=2)
            assert np.all(err[nrm == 0] == 0)
            assert np.all(err <= 1e-2 * nrm), (l, e, float((err / np.maximum(nrm, 1e-30)).max()))


def test_dense_ragged_episodes():
    # g = 64: one K block per group; k from 0 to 16, empty kinds, a
    # single-token segment, more than 128 pairs of one group
    E = synth.Episode
    eps = [E(130, 20, 64, 4, 16), E(9, 3, 5, 2, 1), E(0, 6, 3, 3, 3), E(33, 0, 70, 16, 0),
           E(40, 9, 9, 15, 1, n_prop=3, n_act=8)]
    wl = synth.Workload("dense_edge", "bf16", L=2, H=8, dh=128, G=16, C=8, F=32, episodes=tuple(eps), seed=41)
    _run(wl, [(l, e) for l in range(2) for e in range(len(eps))])


def test_dense_g128_several_chunks():
    # g = 128 (N tile 128 in the z GEMM, two K blocks per group) and more
    # than 4096 rows per layer: pair lists of two chunks, a ragged last
    # chunk, many 128-row tiles of v~; sampled episodes checked
    E = synth.Episode
    rng = np.random.default_rng(7)
    eps = [E(int(rng.integers(120, 300)), int(rng.integers(8, 40)), 4, int(rng.choice([2, 4, 8])),
             int(rng.choice([1, 4, 16]))) for _ in range(22)]
    eps[3] = E(200, 10, 4, 0, 0)        # nothing kept
    wl = synth.Workload("dense_chunks", "bf16", L=1, H=16, dh=128, G=16, C=8, F=32, episodes=tuple(eps),
                        seed=43)
    assert sum(e.n_cache for e in eps) > 4096
    _run(wl, [(0, e) for e in (0, 3, 11, 21)])


def test_dense_oft_layer():
    wl = synth.c1()
    _run(wl, [(0, 0)])


@pytest.mark.slow
def test_dense_c4_full_size_sampled():
    # the bench's workload and launch configuration: 64 ragged episodes x 32
    # layers, d = 4096, g = 256 (three pair-list chunks and 91 row tiles of
    # v~ per layer); sampled (layer, episode) pairs, the largest and the
    # smallest episode included
    wl = synth.c4()
    sizes = [ep.n_cache for ep in wl.episodes]
    e_big, e_small = int(np.argmax(sizes)), int(np.argmin(sizes))
    _run(wl, [(0, e_big), (31, e_small), (17, 5), (5, 40)])


def test_dense_g512_two_column_tiles():
    # d = 8192 (64 heads), g = 512: every 128-pair tile of the z GEMM runs as
    # two 256-column tiles, and a group is eight K blocks of the v~ GEMM
    E = synth.Episode
    eps = [E(40, 8, 4, 4, 16), E(7, 3, 3, 2, 1), E(0, 5, 2, 15, 3)]
    wl = synth.Workload("dense_g512", "bf16", L=1, H=64, dh=128, G=16, C=8, F=32, episodes=tuple(eps), seed=47)
    _run(wl, [(0, e) for e in range(len(eps))])
