"""CPU tests of libframefb's host side: exports, frame construction, support
sampling and plans, checked bit for bit (indices) against the oracle."""
import os
import re

import numpy as np
import pytest

from oracle import adapter, frames, support
from paper_2608_26430_gb300 import framefb as ffb

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built_library():
    from paper_2608_26430_gb300.build import build
    build()


def header_functions():
    txt = open(os.path.join(ROOT, "include", "framefb.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(framefb_[a-z_0-9]+)\s*\(", txt)))


def test_library_exports_every_declared_function():
    names = header_functions()
    assert len(names) >= 17
    got = ffb.exported_symbols(names)
    assert all(got.values()), [n for n, ok in got.items() if not ok]
    assert ffb.lib().framefb_abi_version() == 2


@pytest.mark.parametrize("d,k,rho,parseval", [(256, 16, 16, True), (768, 16, 48, True), (22, 6, 6, False),
                                              (22, 6, 6, True), (40, 7, 8, True), (64, 8, 8, False),
                                              (1024, 16, 64, True), (46, 10, 10, True),
                                              (64, 32, 2, True), (768, 384, 2, True)])  # rho = 2: dense DFT
def test_frame_build_matches_oracle(d, k, rho, parseval):
    fr = ffb.Frame(d, k, rho, parseval)
    P = frames.real_frame(d, k, rho, parseval)
    pat = frames.structural_pattern(d, k, rho)
    colptr, rowidx, val = frames.csc_from_dense(P, pat)
    rowptr, colidx, rval = frames.csr_from_dense(P, pat)
    g_colptr, g_rowidx, g_val = fr.csc()
    g_rowptr, g_colidx, g_rval = fr.csr()
    assert np.array_equal(g_colptr, colptr) and np.array_equal(g_rowidx, rowidx)
    assert np.array_equal(g_rowptr, rowptr) and np.array_equal(g_colidx, colidx)
    np.testing.assert_allclose(g_val, val, rtol=0, atol=2e-15)
    np.testing.assert_allclose(g_rval, rval, rtol=0, atol=2e-15)
    row0, nrows = frames.group_table(d, k, rho)
    g0, gn = fr.groups()
    assert np.array_equal(g0, row0) and np.array_equal(gn, nrows)
    assert fr.nnz == pat.sum() and fr.ncols == k * rho
    assert fr.A == pytest.approx(frames.frame_bound(d, k, rho), rel=1e-15)
    assert fr.dft_groups == int(k * rho == d)


@pytest.mark.parametrize("d", [4096, 14336, 3072])
def test_frame_build_large_dims_indices(d):
    fr = ffb.Frame(d, 16, d // 16)
    colptr, rowidx, val = fr.csc()
    assert np.array_equal(colptr, 32 * np.arange(d + 1))
    # column c = i*rho + 2r + s covers the coordinates of group r
    rho = d // 16
    c = np.arange(d)
    r = (c % rho) // 2
    np.testing.assert_array_equal(rowidx.reshape(d, 32), 32 * r[:, None] + np.arange(32)[None, :])
    np.testing.assert_allclose(np.abs(val).max(), 0.25, rtol=1e-15)


@pytest.mark.parametrize("d,k,rho,status", [(22, 5, 6, ffb.FRAMEFB_EUNSUPPORTED), (14, 4, 8, ffb.FRAMEFB_EUNSUPPORTED),
                                            (21, 4, 6, ffb.FRAMEFB_EINVAL), (24, 4, 3, ffb.FRAMEFB_EINVAL),
                                            (0, 4, 2, ffb.FRAMEFB_EINVAL), (24, 0, 2, ffb.FRAMEFB_EINVAL)])
def test_frame_build_rejects(d, k, rho, status):
    with pytest.raises(ffb.FramefbError) as e:
        ffb.Frame(d, k, rho)
    assert e.value.status == status


SUPPORT_CASES = [(256, 256, 128, 1, 0, 1), (768, 768, 1000, 1, 0, 1), (4096, 4096, 4096, 1, 0, 1),
                 (4096, 14336, 8192, 1, 1, 1), (1024, 4096, 8192, 1, 1, 1), (14336, 4096, 8192, 1, 1, 1),
                 (768, 768, 2000, 1, 0, 1), (96, 96, 500, 3, 2, 16), (64, 32, 2048, 9, 0, 1), (10, 10, 0, 1, 0, 1)]


@pytest.mark.parametrize("rows,cols,nnz,seed,mode,k", SUPPORT_CASES)
def test_support_build_bit_exact(rows, cols, nnz, seed, mode, k):
    row, col, rowptr, perm = ffb.framefb_support_build(rows, cols, nnz, seed, mode, 1.1, k)
    orow, ocol, orowptr, operm = support.sample_support(rows, cols, nnz, seed, mode, 1.1, k)
    assert np.array_equal(row, orow) and np.array_equal(col, ocol)
    assert np.array_equal(rowptr, orowptr) and np.array_equal(perm, operm)


def test_support_build_rejects():
    for args in [(10, 10, 101, 1, 0, 1.1, 1), (10, 10, 5, 1, 7, 1.1, 1), (10, 12, 5, 1, 2, 1.1, 3),
                 (10, 10, 5, 1, 1, -1.0, 1), (0, 10, 0, 1, 0, 1.1, 1)]:
        with pytest.raises(ffb.FramefbError) as e:
            ffb.framefb_support_build(*args)
        assert e.value.status == ffb.FRAMEFB_EINVAL


# ---------------------------------------------------------------------------
# plans: decode the image and replay the kernels' sparse steps on the CPU
# ---------------------------------------------------------------------------
HDR = ["magic", "version", "n", "m", "Gn", "Gm", "nnz", "P", "EZ", "EG", "ovfZ", "ovfG", "nfixZ", "nfixG",
       "off_zb", "off_zq", "off_ga", "off_gb", "off_gq", "off_fixZ", "off_fixG", "off_zmask", "off_gmask",
       "off_blkptr", "off_blkent", "total_bytes", "layout", "d_in", "d_out", "nnz_full", "off_qlist"]


def decode(img):
    h = dict(zip(HDR, np.frombuffer(img[:4 * len(HDR)].tobytes(), dtype=np.int32).tolist()))
    def arr(off, count, dt=np.int32):
        return np.frombuffer(img[off:off + count * np.dtype(dt).itemsize].tobytes(), dtype=dt)
    P = h["P"]
    t = dict(h=h)
    t["zb"] = arr(h["off_zb"], h["EZ"] * P, np.uint32).reshape(h["EZ"], P)
    t["zq"] = arr(h["off_zq"], h["EZ"] * P).reshape(h["EZ"], P)
    t["ga"] = arr(h["off_ga"], h["EG"] * P, np.uint32).reshape(h["EG"], P)
    t["gb"] = arr(h["off_gb"], h["EG"] * P, np.uint32).reshape(h["EG"], P)
    t["gq"] = arr(h["off_gq"], h["EG"] * P).reshape(h["EG"], P)
    t["fixZ"] = arr(h["off_fixZ"], 4 * h["nfixZ"]).reshape(-1, 4)
    t["fixG"] = arr(h["off_fixG"], 4 * h["nfixG"]).reshape(-1, 4)
    t["zmask"] = arr(h["off_zmask"], h["Gm"], np.uint32)
    t["gmask"] = arr(h["off_gmask"], h["Gn"], np.uint32)
    nblk = h["Gm"] * h["Gn"]
    t["blkptr"] = arr(h["off_blkptr"], nblk + 1)
    t["blkent"] = arr(h["off_blkent"], 2 * h["nnz"]).reshape(-1, 2)
    return t


def group_major(c, rho):
    """paper column c = i*rho + 2r + s  ->  x = 32 r + 2 i + s (k = 16)."""
    c = np.asarray(c)
    i, rr = c // rho, c % rho
    return 32 * (rr // 2) + 2 * i + (rr & 1)


def slot(x, K):
    """Tile-buffer slot of group-major index x (the map documented in plan_layout.h)."""
    x = np.asarray(x)
    r, p = x >> 5, (x >> 1) & 15
    pp = p ^ (((p >> 3) & 1) << 1) ^ (r & 1) ^ ((r & 1) << 3)
    return np.where(x >= K, x, (r << 5) | (pp << 1) | (x & 1))


def test_slot_map_is_a_pair_preserving_bijection_and_bank_spread():
    K = 4096
    s = slot(np.arange(K), K)
    assert sorted(s.tolist()) == list(range(K))
    assert np.all(s >> 5 == np.arange(K) >> 5)            # stays inside its group
    assert np.all((s[0::2] ^ 1) == s[1::2])               # pairs stay adjacent, even first
    # the MMA prologue / epilogue: lane (g, t) touches pair 4t + k of group G0 + g;
    # a quarter-warp (g in {0, 1}, t in 0..3) must hit 8 distinct 16-byte bank groups
    # in the two-token layout (one 16-byte chunk per pair)
    for G0 in range(0, 64, 2):
        for k in range(4):
            chunks = [(slot(32 * (G0 + g) + 2 * (4 * t + k), K) >> 1) % 8 for g in (0, 1) for t in range(4)]
            assert len(set(chunks)) == 8
    # one-token layout (a 16-byte chunk holds two pairs): lane (g, t) touches
    # chunk q = 2t + h of group G0 + g; a quarter-warp (g in {0, 1}) must hit
    # 8 distinct 16-byte positions of the 128-byte line
    for G0 in range(0, 64, 2):
        for h in range(2):
            chunks = [(slot(32 * (G0 + g) + 4 * (2 * t + h), K) >> 2) % 8 for g in (0, 1) for t in range(4)]
            assert len(set(chunks)) == 8


PLAN_CASES = [(256, 256, 128, 0), (768, 768, 1000, 0), (768, 3072, 2000, 0), (4096, 1024, 8192, 1),
              (1024, 256, 6000, 1), (256, 768, 4000, 0), (512, 512, 7, 0), (256, 256, 256 * 17, 0),
              (768, 768, 1000, 2), (3072, 768, 2000, 2)]


# frames outside the structured kernels: plans cut for the dense path, whose
# index space is the paper's column order (rho = 2 frames, T-block frames)
DENSE_PLAN_CASES = [((768, 384, 2), (768, 384, 2), 1000, 0), ((4096, 2048, 2), (1024, 512, 2), 8192, 1),
                    ((40, 7, 8), (22, 6, 6), 200, 0), ((46, 10, 10), (46, 10, 10), 2000, 1),
                    ((256, 16, 16), (22, 6, 6), 300, 0)]


@pytest.mark.parametrize("n,m,nnz,mode", PLAN_CASES + DENSE_PLAN_CASES)
def test_plan_replays_coefficient_products(n, m, nnz, mode):
    pin = n if isinstance(n, tuple) else (n, 16, n // 16)
    pout = m if isinstance(m, tuple) else (m, 16, m // 16)
    fin, fout = ffb.Frame(*pin), ffb.Frame(*pout)
    structured = fin.structured and fout.structured
    n, m = pin[1] * pin[2], pout[1] * pout[2]  # index spaces K_n, K_m
    row, col, _, _ = support.sample_support(m, n, nnz, 1, mode, 1.1, 16)  # k: the diagonal blocks of mode 2
    t = decode(ffb.Plan(fin, fout, row, col).image())
    h = t["h"]
    assert h["magic"] == 0x50424646 and h["P"] == ffb.THREADS and h["nnz"] == nnz
    assert h["layout"] == (0 if structured else 1) and (h["n"], h["m"]) == (n, m)
    assert (h["d_in"], h["d_out"]) == (pin[0], pout[0])
    # every entry appears once in each chunk table
    assert sorted(t["zq"][t["zq"] >= 0].tolist()) == list(range(nnz))
    assert sorted(t["gq"][t["gq"] >= 0].tolist()) == list(range(nnz))
    if structured:
        a_int, b_int = group_major(row, m // 16), group_major(col, n // 16)
    else:
        a_int, b_int = np.asarray(row), np.asarray(col)
    assert len(set(a_int.tolist())) == len(set(row.tolist()))
    # masks
    zm = np.zeros(h["Gm"], np.uint32)
    gm = np.zeros(h["Gn"], np.uint32)
    for a in a_int:
        zm[a >> 5] |= np.uint32(1) << np.uint32(a & 31)
    for b in b_int:
        gm[b >> 5] |= np.uint32(1) << np.uint32(b & 31)
    assert np.array_equal(zm, t["zmask"]) and np.array_equal(gm, t["gmask"])

    # replay with random V (input side) and U (output side) rows, 3 tokens
    rng = np.random.default_rng(0)
    Tn = 3
    c = rng.standard_normal(nnz)
    Vint = rng.standard_normal((Tn, n))
    Uint = rng.standard_normal((Tn, m))
    Vs, Us = Vint, Uint                  # the tables hold group-major indices
    RZ = np.zeros((Tn, m + h["ovfZ"]))
    RG = np.zeros((Tn, n + h["ovfG"]))
    dC = np.zeros(nnz)
    for p in range(h["P"]):
        acc = np.zeros(Tn)
        for e in range(h["EZ"]):
            pk, q = int(t["zb"][e, p]), int(t["zq"][e, p])
            cv = c[q] if q >= 0 else 0.0
            if q >= 0:  # bit 15 carries the parity of the entry's row
                assert (pk >> 15) & 1 == a_int[q] & 1
            acc += cv * Vs[:, pk & 0x7FFF]
            if (pk >> 16) != 0xFFFF:
                RZ[:, pk >> 16] = acc
                acc = np.zeros(Tn)
        acc = np.zeros(Tn)
        for e in range(h["EG"]):
            pa, pb, q = int(t["ga"][e, p]), int(t["gb"][e, p]), int(t["gq"][e, p])
            cv = c[q] if q >= 0 else 0.0
            if q >= 0:  # bit 15 carries the parity of the entry's column
                assert (pa >> 15) & 1 == b_int[q] & 1
            uv = Us[:, pa & 0x7FFF]
            acc += cv * uv
            if q >= 0:
                dC[q] += np.dot(uv, Vs[:, pb])
            if (pa >> 16) != 0xFFFF:
                RG[:, pa >> 16] = acc
                acc = np.zeros(Tn)
    for dst, src, cnt, _ in t["fixZ"]:
        RZ[:, dst] += RZ[:, src:src + cnt].sum(axis=1)
    for dst, src, cnt, _ in t["fixG"]:
        RG[:, dst] += RG[:, src:src + cnt].sum(axis=1)
    Z = RZ[:, :m]
    G = RG[:, :n]
    Cint = adapter.dense_C(m, n, a_int, b_int, c)
    np.testing.assert_allclose(Z, Vint @ Cint.T, atol=1e-12)
    np.testing.assert_allclose(G, Uint @ Cint, atol=1e-12)
    np.testing.assert_allclose(dC, np.einsum("ta,tb->ab", Uint, Vint)[a_int, b_int], atol=1e-12)
    # merge blocks list every entry once with its local indices
    seen = []
    Gn = h["Gn"]
    for blk in range(h["Gm"] * Gn):
        for e in range(t["blkptr"][blk], t["blkptr"][blk + 1]):
            pk, q = t["blkent"][e]
            g, hh = divmod(blk, Gn)
            assert 32 * g + (pk & 31) == a_int[q] and 32 * hh + ((pk >> 8) & 31) == b_int[q]
            seen.append(int(q))
    assert sorted(seen) == list(range(nnz))


def test_plan_rejects_unsorted_and_unsupported():
    f256 = ffb.Frame(256, 16, 16)
    with pytest.raises(ffb.FramefbError) as e:
        ffb.Plan(f256, f256, np.array([3, 1], np.int32), np.array([0, 0], np.int32))
    assert e.value.status == ffb.FRAMEFB_EINVAL
    with pytest.raises(ffb.FramefbError) as e:
        ffb.Plan(f256, f256, np.array([1, 1], np.int32), np.array([2, 2], np.int32))
    assert e.value.status == ffb.FRAMEFB_EINVAL
    with pytest.raises(ffb.FramefbError) as e:
        ffb.Plan(f256, f256, np.array([256], np.int32), np.array([0], np.int32))
    assert e.value.status == ffb.FRAMEFB_EINVAL
    # T-block and rho = 2 frames get plans cut for the dense path; a mixed
    # pair (one structured frame) does too
    red, dense = ffb.Frame(22, 6, 6), ffb.Frame(64, 32, 2)
    for fi, fo, K in ((red, red, 36), (dense, dense, 64), (f256, red, 36)):
        h = decode(ffb.Plan(fi, fo, np.array([0, 1], np.int32), np.array([0, 3], np.int32)).image())["h"]
        assert h["layout"] == 1 and h["m"] == K
    with pytest.raises(ffb.FramefbError) as e:  # row outside K_m = 36
        ffb.Plan(red, red, np.array([36], np.int32), np.array([0], np.int32))
    assert e.value.status == ffb.FRAMEFB_EINVAL
    p = ffb.Plan(f256, f256, np.zeros(0, np.int32), np.zeros(0, np.int32))
    assert decode(p.image())["h"]["nnz"] == 0


@pytest.mark.parametrize("d,k,rho", [(22, 6, 6), (40, 7, 8), (64, 32, 2), (768, 384, 2), (256, 16, 16)])
def test_dense_operand_image_matches_oracle_frame(d, k, rho):
    """framefb_frame_dense_pack against the oracle's dense frame: the bf16
    hi + lo analysis operand (rows = columns of Phi) carries Phi to 2^-16
    relative, the synthesis operand (rows = rows of Phi) is Phi rounded to
    tf32, and padding is zero."""
    f = ffb.Frame(d, k, rho)
    P = frames.real_frame(d, k, rho, parseval=True)
    K = k * rho
    img = f.dense_image()
    dp, cp = -(-d // 8) * 8, -(-K // 4) * 4
    an = -(-(K * dp * 2) // 1024) * 1024
    assert img.size == 2 * an + -(-(d * cp * 4) // 1024) * 1024

    def bf16(words):
        return (np.asarray(words, np.uint32) << 16).view(np.float32).astype(np.float64)
    hi = bf16(img[:K * dp * 2].view(np.uint16)).reshape(K, dp)
    lo = bf16(img[an:an + K * dp * 2].view(np.uint16)).reshape(K, dp)
    sy = img[2 * an:2 * an + d * cp * 4].view(np.float32).astype(np.float64).reshape(d, cp)
    amax = np.abs(P).max()
    assert np.max(np.abs(hi[:, :d] + lo[:, :d] - P.T)) <= 2.0 ** -16 * amax
    assert np.max(np.abs(hi[:, :d] - P.T)) <= 2.0 ** -8 * amax             # hi is the bf16 rounding
    assert np.max(np.abs(sy[:, :K] - P)) <= 2.0 ** -11 * amax                # tf32 rounding
    assert not hi[:, d:].any() and not lo[:, d:].any() and not sy[:, K:].any()
    bits = img[2 * an:2 * an + d * cp * 4].view(np.uint32)
    assert np.all(bits & 0x1FFF == 0)                                        # 10-bit mantissas


# ---------------------------------------------------------------------------
# parts: plans the fused tcgen05 kernels cannot take whole (LLaMA-3 shapes)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("n,m,nnz,mode", [(4096, 14336, 8192, 1), (14336, 4096, 8192, 1), (4096, 4096, 8192, 1),
                                          (4096, 1024, 8192, 1), (4096, 4096, 4096 * 2 + 5, 0),
                                          (14336, 14336, 9000, 0), (4096, 4096, 4096, 1)])
def test_plan_parts_cover_the_support_once(n, m, nnz, mode):
    fin, fout = ffb.Frame(n, 16, n // 16), ffb.Frame(m, 16, m // 16)
    row, col, _, _ = support.sample_support(m, n, nnz, 1, mode, 1.1, 16)
    plan = ffb.Plan(fin, fout, row, col)
    img = plan.image()
    parts = plan.parts()
    whole = decode(img)["h"]
    if (whole["EZ"] <= 16 and whole["Gm"] <= 128) or whole["Gn"] > 128:
        assert parts == []      # the fused kernels take it whole, or input blocks would be needed
        return
    assert all(pt["n0"] == 0 and pt["n"] == n for pt in parts)
    assert parts and whole["total_bytes"] <= parts[0]["image_offset"]
    a_gm, b_gm = group_major(row, m // 16), group_major(col, n // 16)
    seen = np.zeros(nnz, np.int32)
    for pt in parts:
        off = pt["image_offset"]
        assert off % 256 == 0 and off + pt["image_bytes"] <= img.size
        t = decode(img[off:off + pt["image_bytes"]])
        h = t["h"]
        # a plan of its own within the kernels' limits, over whole groups
        assert (h["n"], h["m"], h["nnz"]) == (pt["n"], pt["m"], pt["nnz"]) and h["nnz_full"] == nnz
        assert h["EZ"] <= 16 and h["EG"] <= 16 and h["nnz"] <= 16 * ffb.THREADS
        assert h["Gn"] <= 128 and h["Gm"] <= 128 and h["Gn"] % 8 == 0 and h["Gm"] % 8 == 0
        assert pt["n0"] % 256 == 0 and pt["m0"] % 256 == 0 and pt["n0"] + pt["n"] <= n and pt["m0"] + pt["m"] <= m
        assert (h["d_in"], h["d_out"]) == (n, m)
        # its entry list, in its own image and at q_offset of the parent's
        q = np.frombuffer(img[off + h["off_qlist"]:off + h["off_qlist"] + 4 * h["nnz"]].tobytes(), np.int32)
        q2 = np.frombuffer(img[pt["q_offset"]:pt["q_offset"] + 4 * pt["nnz"]].tobytes(), np.int32)
        assert np.array_equal(q, q2)
        seen[q] += 1
        assert sorted(t["zq"][t["zq"] >= 0].tolist()) == sorted(q.tolist())
        assert sorted(t["gq"][t["gq"] >= 0].tolist()) == sorted(q.tolist())
        # block lists: every entry's local (a, b) is its group-major index less the blocks' start
        for blk in range(h["Gm"] * h["Gn"]):
            g, hh = divmod(blk, h["Gn"])
            for e in range(t["blkptr"][blk], t["blkptr"][blk + 1]):
                x, qq = t["blkent"][e]
                assert 32 * g + (x & 31) == a_gm[qq] - pt["m0"]
                assert 32 * hh + ((x >> 8) & 31) == b_gm[qq] - pt["n0"]
    assert np.all(seen == 1)     # every entry in exactly one part


@pytest.mark.parametrize("n,m", [(4096, 14336), (4096, 4096)])
def test_plan_parts_replay_coefficient_products(n, m):
    """Every part of a Zipf(1.1) LLaMA-3-shaped plan (8192 entries) replays
    the kernels' sparse steps exactly: run sums by row and by column with the
    overflow slots and fix-ups, and the dC products, against the part's
    entries at their block-local indices."""
    nnz = 8192
    fin, fout = ffb.Frame(n, 16, n // 16), ffb.Frame(m, 16, m // 16)
    row, col, _, _ = support.sample_support(m, n, nnz, 1, 1, 1.1, 16)
    plan = ffb.Plan(fin, fout, row, col)
    img, parts = plan.image(), plan.parts()
    assert parts
    a_gm, b_gm = group_major(row, m // 16), group_major(col, n // 16)
    rng = np.random.default_rng(1)
    c = rng.standard_normal(nnz)
    for pt in parts:
        off = pt["image_offset"]
        t = decode(img[off:off + pt["image_bytes"]])
        h = t["h"]
        nv, mv = h["n"], h["m"]
        V, U = rng.standard_normal((2, nv)), rng.standard_normal((2, mv))
        RZ, RG = np.zeros((2, mv + h["ovfZ"])), np.zeros((2, nv + h["ovfG"]))
        dC = np.zeros(nnz)
        for p in range(h["P"]):
            acc = np.zeros(2)
            for e in range(h["EZ"]):
                pk, q = int(t["zb"][e, p]), int(t["zq"][e, p])
                acc += (c[q] if q >= 0 else 0.0) * V[:, pk & 0x7FFF]
                if (pk >> 16) != 0xFFFF:
                    RZ[:, pk >> 16] = acc
                    acc = np.zeros(2)
            acc = np.zeros(2)
            for e in range(h["EG"]):
                pa, pb, q = int(t["ga"][e, p]), int(t["gb"][e, p]), int(t["gq"][e, p])
                acc += (c[q] if q >= 0 else 0.0) * U[:, pa & 0x7FFF]
                if q >= 0:
                    dC[q] += U[:, pa & 0x7FFF] @ V[:, pb]
                if (pa >> 16) != 0xFFFF:
                    RG[:, pa >> 16] = acc
                    acc = np.zeros(2)
        for dst, src, cnt, _ in t["fixZ"]:
            RZ[:, dst] += RZ[:, src:src + cnt].sum(axis=1)
        for dst, src, cnt, _ in t["fixG"]:
            RG[:, dst] += RG[:, src:src + cnt].sum(axis=1)
        q = np.frombuffer(img[pt["q_offset"]:pt["q_offset"] + 4 * pt["nnz"]].tobytes(), np.int32)
        al, bl = a_gm[q] - pt["m0"], b_gm[q] - pt["n0"]
        Cl = adapter.dense_C(mv, nv, al, bl, c[q])
        np.testing.assert_allclose(RZ[:, :mv], V @ Cl.T, atol=1e-12)
        np.testing.assert_allclose(RG[:, :nv], U @ Cl, atol=1e-12)
        np.testing.assert_allclose(dC[q], np.einsum("ta,tb->ab", U, V)[al, bl], atol=1e-12)
        assert not np.any(np.delete(dC, q))      # a part writes only its own entries
