"""C-ABI checks that need no GPU: the library loads, exports every function
include/rolesub.h declares, plans the cache layout exactly like the oracle's
independent layout code, reproduces the paper's KV accounting, and rejects
bad arguments before touching the device."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2608_18410_gb300 import build as pkg_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def rsm():
    pkg_build.build()
    from paper_2608_18410_gb300 import rolesub
    rolesub.lib()
    return rolesub


def declared_functions():
    txt = open(os.path.join(ROOT, "include", "rolesub.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(rolesub_[a-z_]+)\s*\(", txt)))


def test_header_and_binding_agree(rsm):
    decl = declared_functions()
    assert set(decl) == set(rsm.EXPORTS), decl


def test_every_declared_symbol_is_exported(rsm):
    L = ctypes.CDLL(rsm.LIB_PATH)
    for name in declared_functions():
        assert hasattr(L, name), name
    assert rsm.rolesub_version() == 1
    assert rsm.rolesub_status_string(1) == "invalid argument"


def test_static_scratch_size_matches_header(rsm):
    txt = open(os.path.join(ROOT, "include", "rolesub.h")).read()
    m = re.search(r"#define ROLESUB_STATIC_SCRATCH_BYTES \((\d+)u << (\d+)\)", txt)
    assert m, "ROLESUB_STATIC_SCRATCH_BYTES not found in the header"
    assert rsm.rolesub_static_scratch_bytes() == int(m.group(1)) << int(m.group(2))


def test_struct_sizes_match_header(rsm):
    assert ctypes.sizeof(rsm.Shape) == 32
    assert ctypes.sizeof(rsm.Segment) == 40
    assert ctypes.sizeof(rsm.Episode) == 40
    assert ctypes.sizeof(rsm.PlanHeader) == 152


def _plan(rsm, n_tok, k, n_q, H=2, dh=8, G=4, dtype="f32"):
    shape = rsm.make_shape(1, H, dh, G, 3, 8, dtype)
    return rsm.Plan(shape, n_tok, k, n_q)


def test_plan_matches_oracle_layout(rsm, oracle):
    rng = np.random.default_rng(0)
    for trial in range(20):
        E = int(rng.integers(0, 6))
        H, dh, G = [(2, 8, 4), (32, 128, 16), (8, 64, 8), (3, 16, 1)][trial % 4]
        n_tok = rng.integers(0, 40, size=(E, 4)).astype(np.int32)
        k = rng.integers(0, G + 1, size=(E, 4)).astype(np.int32)
        n_q = rng.integers(0, 70, size=E).astype(np.int32)
        p = _plan(rsm, n_tok, k, n_q, H, dh, G)
        ref = oracle.layout(n_tok, k, H, dh, G) if E else {"rows": 0, "packed_elems": 0, "idx_bytes": 0}
        assert p.hdr.rows_per_layer == ref["rows"]
        assert p.hdr.packed_elems_per_layer == ref["packed_elems"]
        assert p.hdr.idx_bytes_per_layer == ref["idx_bytes"]
        assert p.hdr.q_rows_per_layer == int(n_q.sum())
        for s, seg in enumerate(p.segments):
            assert (seg.episode, seg.kind) == (s // 4, s % 4)
            assert seg.n_tokens == n_tok.reshape(-1)[s] and seg.k == k.reshape(-1)[s]
            assert seg.token_row == ref["row_off"][s]
            assert seg.packed_off == ref["packed_off"][s]
            assert seg.idx_off == ref["idx_off"][s]
        routed = sum(int(n_tok.reshape(-1)[s]) for s in range(4 * E) if 0 < k.reshape(-1)[s] < G)
        stored = sum(int(n_tok.reshape(-1)[s]) for s in range(4 * E) if k.reshape(-1)[s] > 0)
        assert p.hdr.routed_rows_per_layer == routed
        assert p.hdr.stored_rows_per_layer == stored
        # routed / stored row lists
        h = p.hdr
        rr = np.frombuffer(p.host[h.off_routed_rows:h.off_routed_rows + 4 * routed].tobytes(), np.int32)
        sr = np.frombuffer(p.host[h.off_stored_rows:h.off_stored_rows + 4 * stored].tobytes(), np.int32)
        rs_ = np.frombuffer(p.host[h.off_row_seg:h.off_row_seg + 4 * h.rows_per_layer].tobytes(), np.int32)
        kk = k.reshape(-1)
        assert np.all(np.diff(rr) > 0) and np.all(np.diff(sr) > 0)
        assert all(0 < kk[rs_[r]] < G for r in rr) and all(kk[rs_[r]] > 0 for r in sr)
        for s, seg in enumerate(p.segments):
            assert np.all(rs_[seg.token_row:seg.token_row + seg.n_tokens] == s)
        # router tiles: 128-row windows that start on routed rows and cover
        # every routed row exactly once
        nt = h.num_route_tiles
        tiles = np.frombuffer(p.host[h.off_route_tiles:h.off_route_tiles + 4 * nt].tobytes(), np.int32)
        assert np.all(np.isin(tiles, rr)) and np.all(np.diff(tiles) >= 128)
        cover = np.zeros(h.rows_per_layer, int)
        for t0 in tiles:
            cover[t0:t0 + 128] += 1
        assert np.all(cover[rr] == 1)


def test_plan_reproduces_table_1_visual_kv(rsm):
    import math
    H, dh, G = 32, 128, 16
    d = H * dh
    for n_keep, K, pct in [(8, 1, 0.83), (8, 2, 0.88), (8, 4, 0.98), (16, 1, 1.66), (16, 2, 1.76),
                           (16, 4, 1.95), (32, 1, 3.32), (32, 2, 3.52), (32, 4, 3.91)]:
        p = _plan(rsm, [[n_keep, 0, 0, 0]], [[K, G, G, G]], [8], H, dh, G, "bf16")
        kv = (n_keep * d + p.hdr.packed_elems_per_layer) / (2.0 * 512 * d)
        assert math.floor(100 * kv * 100 + 0.5 + 1e-9) / 100 == pytest.approx(pct)


def test_plan_rejects_bad_arguments(rsm):
    with pytest.raises(rsm.RoleSubError):
        _plan(rsm, [[3, 0, 0, 0]], [[5, 4, 4, 4]], [1])          # k > S
    with pytest.raises(rsm.RoleSubError):
        _plan(rsm, [[-1, 0, 0, 0]], [[2, 4, 4, 4]], [1])         # negative count
    for bad in [dict(G=3), dict(G=17, dh=34), dict(dh=0)]:
        kw = dict(H=2, dh=8, G=4)
        kw.update(bad)
        with pytest.raises(rsm.RoleSubError):
            _plan(rsm, [[3, 0, 0, 0]], [[2, 4, 4, 4]], [1], **kw)


def test_calls_reject_bad_arguments_before_any_launch(rsm):
    shape = rsm.make_shape(1, 2, 8, 4, 3, 8, "f32")
    plan = rsm.Plan(shape, [[3, 0, 0, 0]], [[2, 4, 4, 4]], [1])
    L = rsm.lib()
    fake = 1 << 20    # never dereferenced: validation fails first
    args = [ctypes.byref(shape), plan.host_ptr, fake] + [fake] * 9 + [0.1, 0.1, fake, fake, fake, 1 << 30, None]
    # null h
    a = list(args)
    a[3] = None
    assert L.rolesub_compress(*a) == 1
    # unaligned v
    a = list(args)
    a[4] = fake + 2
    assert L.rolesub_compress(*a) == 1
    # workspace too small
    a = list(args)
    a[17] = 16
    assert L.rolesub_compress(*a) == 1
    # non-finite alpha
    a = list(args)
    a[12] = float("nan")
    assert L.rolesub_compress(*a) == 1
    # plan for another geometry
    other = rsm.make_shape(1, 2, 16, 4, 3, 8, "f32")
    a = list(args)
    a[0] = ctypes.byref(other)
    assert L.rolesub_compress(*a) == 1
    # corrupted plan magic
    bad = plan.host.copy()
    bad[0] ^= 0xFF
    a = list(args)
    a[1] = bad.ctypes.data
    assert L.rolesub_compress(*a) == 1
    # attend: stride not a multiple of 16 bytes
    at = [ctypes.byref(shape), plan.host_ptr, fake, fake, 8 * 16, 16, 3, fake, 8 * 16, 16, 8, fake, fake,
          fake, 0.0, fake, fake, 1 << 30, None]
    assert L.rolesub_attend(*at) == 1
    at[6] = 8
    at[14] = -1.0                                                # negative scale
    assert L.rolesub_attend(*at) == 1
    # unsupported head_dim for this build (valid geometry otherwise)
    s2 = rsm.make_shape(1, 2, 40, 4, 3, 8, "f32")
    p2 = rsm.Plan(s2, [[3, 0, 0, 0]], [[2, 4, 4, 4]], [1])
    at2 = [ctypes.byref(s2), p2.host_ptr, fake, fake, 80 * 16, 80, 40, fake, 80 * 16, 80, 40, fake, fake,
           fake, 0.0, fake, fake, 1 << 30, None]
    assert L.rolesub_attend(*at2) == 2


def test_additive_compress_rejects_bad_arguments_before_any_launch(rsm):
    shape = rsm.make_shape(1, 2, 8, 4, 3, 8, "f32")
    plan = rsm.Plan(shape, [[3, 2, 0, 0]], [[2, 4, 4, 4]], [1])
    L = rsm.lib()
    fake = 1 << 20    # never dereferenced: validation fails first
    # shape, plan, plan_dev, h v R W_re b_re W_v b_v W_role W_l b_l, alphas, packed idx ws ws_bytes stream
    args = [ctypes.byref(shape), plan.host_ptr, fake] + [fake] * 10 + [0.1, 0.1, fake, fake, fake, 1 << 30, None]
    for pos in range(3, 13):          # every weight or input pointer null
        a = list(args)
        a[pos] = None
        assert L.rolesub_compress_additive(*a) == 1, pos
    a = list(args)
    a[9] = fake + 4                   # b_v not 16-byte aligned
    assert L.rolesub_compress_additive(*a) == 1
    a = list(args)
    a[13] = float("inf")
    assert L.rolesub_compress_additive(*a) == 1
    a = list(args)
    a[18] = 16                        # workspace too small
    assert L.rolesub_compress_additive(*a) == 1
    # more role components than the fallback's shared-memory scratch holds
    big = rsm.make_shape(1, 2, 8, 4, 5000, 8, "f32")
    pb = rsm.Plan(big, [[3, 2, 0, 0]], [[2, 4, 4, 4]], [1])
    a = list(args)
    a[0], a[1] = ctypes.byref(big), pb.host_ptr
    assert L.rolesub_compress_additive(*a) == 2


def test_budget_calls_reject_bad_arguments_before_any_launch(rsm):
    shape = rsm.make_shape(1, 2, 128, 16, 6, 8, "bf16")
    plan = rsm.Plan(shape, [[3, 2, 0, 0]], [[4, 16, 16, 16]], [1])
    L = rsm.lib()
    fake = 1 << 20    # never dereferenced: validation fails first
    big = plan.budget_workspace_size()
    assert big > plan.workspace_size()
    # shape, plan, plan_dev, h v R W_re b_re W_v b_v W_role W_l b_l u, alphas, packed idx k_tok ws, ws_bytes, stream
    args = [ctypes.byref(shape), plan.host_ptr, fake] + [fake] * 11 + [0.1, 0.1, fake, fake, fake, fake, big, None]
    for pos in range(3, 14):
        a = list(args)
        a[pos] = None
        assert L.rolesub_compress_budget(*a) == 1, pos
    a = list(args)
    a[18] = None                      # k_tok
    assert L.rolesub_compress_budget(*a) == 1
    a = list(args)
    a[20] = big - 16                  # workspace without room for the scores
    assert L.rolesub_compress_budget(*a) == 1
    f32 = rsm.make_shape(1, 2, 64, 8, 6, 8, "f32")
    p32 = rsm.Plan(f32, [[3, 2, 0, 0]], [[4, 8, 8, 8]], [1])
    a = list(args)
    a[0], a[1] = ctypes.byref(f32), p32.host_ptr
    assert L.rolesub_compress_budget(*a) == 2   # the budget path is bf16, d_h = 128, S = 16 only
    at = [ctypes.byref(shape), plan.host_ptr, fake, fake, 0, 2048, 128, fake, 0, 2048, 128, fake, fake, None,
          fake, 0.0, fake, fake, 1 << 30, None]
    assert L.rolesub_attend_budget(*at) == 1    # no k_tok
    at[13] = fake
    at[0], at[1] = ctypes.byref(f32), p32.host_ptr
    at[5], at[6], at[9], at[10] = 1024, 64, 1024, 64
    assert L.rolesub_attend_budget(*at) == 2


def test_select_tokens_rejects_bad_arguments_before_any_launch(rsm):
    L = rsm.lib()
    fake = 1 << 20
    assert L.rolesub_select_count(256, 0.0625) == 16
    assert L.rolesub_select_count(300, 0.0625) == 19
    assert L.rolesub_select_count(8, 0.0) == -1
    assert L.rolesub_select_tokens(1, 2, 8, 0.0, fake, fake, 8, 0, fake, fake, None) == 1       # ratio 0
    assert L.rolesub_select_tokens(1, 2, 8, 0.5, fake, fake, 3, 0, fake, fake, None) == 1       # 12-byte rows
    assert L.rolesub_select_tokens(1, 2, 8, 0.5, fake + 4, fake, 8, 0, fake, fake, None) == 1   # unaligned
    assert L.rolesub_select_tokens(1, 2, 20000, 0.5, fake, fake, 8, 0, fake, fake, None) == 1   # n_view too big
    assert L.rolesub_select_tokens(0, 2, 8, 0.5, None, None, 8, 0, None, None, None) == 0       # nothing to do


def test_dense_calls_reject_bad_arguments_before_any_launch(rsm):
    shape = rsm.make_shape(1, 8, 128, 16, 8, 32, "bf16")   # d = 1024, g = 64
    plan = rsm.Plan(shape, [[3, 2, 0, 0]], [[4, 16, 16, 16]], [1])
    L = rsm.lib()
    fake = 1 << 20
    big = plan.dense_workspace_size()
    assert big > plan.workspace_size()
    # shape, plan, plan_dev, h v R_dense W_re b_re W1 b1 W2 b2, alphas, packed idx ws, ws_bytes, stream
    args = [ctypes.byref(shape), plan.host_ptr, fake] + [fake] * 9 + [0.1, 0.1, fake, fake, fake, big, None]
    for pos in range(3, 12):
        a = list(args)
        a[pos] = None
        assert L.rolesub_compress_dense(*a) == 1, pos
    a = list(args)
    a[17] = big - 256                   # workspace without the dense buffers
    assert L.rolesub_compress_dense(*a) == 1
    for H in (3, 4, 6):
        # d = 384 (not a multiple of 256), g = 32 (less than a 64-wide K
        # block), g = 48: unsupported group geometry
        odd = rsm.make_shape(1, H, 128, 16, 8, 32, "bf16")
        po = rsm.Plan(odd, [[3, 2, 0, 0]], [[4, 16, 16, 16]], [1])
        a = list(args)
        a[0], a[1] = ctypes.byref(odd), po.host_ptr
        a[17] = po.dense_workspace_size()
        assert L.rolesub_compress_dense(*a) == 2, H
    at = [ctypes.byref(shape), plan.host_ptr, fake, fake, 0, 1024, 128, fake, 0, 1024, 128, fake, fake, fake,
          0.0, fake, fake, big, None]
    at[13] = None                       # R_dense
    assert L.rolesub_attend_dense(*at) == 1
    at[13] = fake
    at[17] = big - 256
    assert L.rolesub_attend_dense(*at) == 1


def test_wait_selftest_rejects_bad_arguments_before_any_launch(rsm):
    L = rsm.lib()
    fake = 1 << 20            # never touched: every check comes before the launch
    assert L.rolesub_wait_selftest(999, fake, fake, None) == 1
    assert L.rolesub_wait_selftest(2_000_000_001, fake, fake, None) == 1
    assert L.rolesub_wait_selftest(5_000_000, None, fake, None) == 1
    assert L.rolesub_wait_selftest(5_000_000, fake, None, None) == 1
    assert L.rolesub_wait_selftest(5_000_000, fake + 8, fake, None) == 1
