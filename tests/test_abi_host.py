"""Host-only checks of the C ABI: the library builds, loads, exports every
entry point include/fbob.h declares, and validates arguments before touching
CUDA (so these run without a GPU)."""
import ctypes

import pytest

import paper_2609_24089_gb300 as fbob


@pytest.fixture(scope="module")
def lib():
    fbob.build()
    return fbob.load()


def test_exports_every_declared_symbol(lib):
    names = fbob.header_symbols()
    assert {"fbob_attn_fwd", "fbob_attn_bwd", "fbob_attn_bob", "fbob_attn_bob_pass1",
            "fbob_attn_bob_pass2", "fbob_attn_bob_row_stats", "fbob_attn_bob_pass1_direct",
            "fbob_device_status", "fbob_status_string", "fbob_launch_count"} <= set(names)
    for n in names:
        assert getattr(lib, n) is not None


def test_status_strings(lib):
    assert lib.fbob_status_string(0) == b"FBOB_OK"
    assert lib.fbob_status_string(2) == b"FBOB_ERR_UNSUPPORTED"
    assert lib.fbob_status_string(99) == b"FBOB_UNKNOWN_STATUS"


# fake, 16-byte aligned, non-overlapping "device" addresses: validation never
# dereferences them, and every call below fails or returns before any CUDA call
BASE = 1 << 40
STRIDE = 1 << 34


def ptrs(n, misalign=None):
    out = [BASE + t * STRIDE for t in range(n)]
    if misalign is not None:
        out[misalign] += 8
    return [ctypes.c_void_p(p) for p in out]


def bob(lib, shape, ps):
    return lib.fbob_attn_bob(ctypes.byref(shape), *ps, None)


def test_rejects_bad_shapes(lib):
    S = fbob.make_shape
    assert bob(lib, S(1, 1, 128, 48, 0.14, 0), ptrs(14)) == 2          # d unsupported
    assert bob(lib, S(1, 1, 128, 16, 0.25, 0), ptrs(14)) == 2
    assert bob(lib, S(1, 1, 128, 512, 0.04, 1), ptrs(14)) == 2
    assert bob(lib, S(1, 1, 128, 96, 0.1, 1), ptrs(14)) == 2
    # d = 256 is supported, except by the one-sweep Pass 1 (four 256-column
    # accumulators do not fit TMEM), which refuses it before any CUDA call
    fused = lib.fbob_attn_bob_pass1_fused
    assert fused(ctypes.byref(S(1, 1, 128, 256, 0.0625, 1)), *ptrs(13), None) == 2
    assert bob(lib, S(1, 1, 128, 64, 0.0, 0), ptrs(14)) == 1           # scale <= 0
    assert bob(lib, S(1, 1, 128, 64, float("nan"), 0), ptrs(14)) == 1
    assert bob(lib, S(1, 1, 128, 64, float("inf"), 0), ptrs(14)) == 1
    assert bob(lib, S(1, 1, 128, 64, 0.125, 2), ptrs(14)) == 1         # causal not 0/1
    assert bob(lib, S(-1, 1, 128, 64, 0.125, 0), ptrs(14)) == 1
    assert bob(lib, S(1, 1, (1 << 24) + 1, 64, 0.125, 0), ptrs(14)) == 1
    # launch grids past 2^31 CTAs: ceil(N/128) * B*H * 2 >= 2^31
    assert bob(lib, S(1 << 12, 1 << 12, 1 << 14, 64, 0.125, 0), ptrs(14)) == 1
    assert lib.fbob_attn_bob(None, *ptrs(14), None) == 1               # null shape


def test_empty_problems_launch_nothing(lib):
    S = fbob.make_shape
    for shp in (S(0, 4, 128, 64, 0.125, 0), S(2, 0, 128, 64, 0.125, 1), S(2, 4, 0, 128, 0.09, 0)):
        assert bob(lib, shp, ptrs(14)) == 0
        assert lib.fbob_launch_count(b"bob") == 0
        assert lib.fbob_attn_fwd(ctypes.byref(shp), *ptrs(5), None) == 0
        assert lib.fbob_attn_bwd(ctypes.byref(shp), *ptrs(10), None) == 0


def test_rejects_null_misaligned_and_overlapping_pointers(lib):
    S = fbob.make_shape(1, 2, 100, 64, 0.125, 1)
    for t in range(14):
        ps = ptrs(14)
        ps[t] = ctypes.c_void_p(0)
        assert bob(lib, S, ps) == 1, t
        assert bob(lib, S, ptrs(14, misalign=t)) == 1, t
    ps = ptrs(14)
    ps[10] = ps[0]                      # k_bar aliases q
    assert bob(lib, S, ps) == 1
    ps = ptrs(14)
    ps[13] = ctypes.c_void_p(ps[12].value + 64)   # row_stats overlaps dout_bar
    assert bob(lib, S, ps) == 1
    # pass 2 reads row_stats: it may not alias its outputs
    ps = ptrs(11)          # q k v lse dout gq gk gv row_stats k_bar v_bar
    ps[9] = ps[8]
    assert lib.fbob_attn_bob_pass2(ctypes.byref(S), *ps, None) == 1


def test_row_stats_and_direct_validate_like_pass1(lib):
    S = fbob.make_shape(1, 2, 100, 128, 0.088, 1)
    rs = lib.fbob_attn_bob_row_stats      # q k v o lse dout gq gk gv row_stats
    pd = lib.fbob_attn_bob_pass1_direct   # q k v lse dout gq gk gv row_stats q_bar dout_bar
    for t in range(10):
        ps = ptrs(10)
        ps[t] = ctypes.c_void_p(0)
        assert rs(ctypes.byref(S), *ps, None) == 1, t
        assert rs(ctypes.byref(S), *ptrs(10, misalign=t), None) == 1, t
    for t in range(11):
        ps = ptrs(11)
        ps[t] = ctypes.c_void_p(0)
        assert pd(ctypes.byref(S), *ps, None) == 1, t
    ps = ptrs(11)
    ps[9] = ps[8]                       # q_bar aliases row_stats (an input here)
    assert pd(ctypes.byref(S), *ps, None) == 1
    bad = fbob.make_shape(1, 2, 100, 96, 0.1, 0)
    assert rs(ctypes.byref(bad), *ptrs(10), None) == 2
    assert pd(ctypes.byref(bad), *ptrs(11), None) == 2
    empty = fbob.make_shape(1, 2, 0, 128, 0.088, 0)
    assert rs(ctypes.byref(empty), *ptrs(10), None) == 0
    assert lib.fbob_launch_count(b"bob_row_stats") == 0
    assert pd(ctypes.byref(empty), *ptrs(11), None) == 0
    assert lib.fbob_launch_count(b"bob_pass1_direct") == 0


def test_rejects_bad_windows(lib):
    S = fbob.make_shape
    assert bob(lib, S(1, 1, 128, 64, 0.125, 0, window=(-2, -1)), ptrs(14)) == 1
    assert bob(lib, S(1, 1, 128, 64, 0.125, 1, window=(3, -5)), ptrs(14)) == 1
    # valid windows pass validation (then stop at the empty problem, no CUDA call)
    assert bob(lib, S(1, 1, 0, 64, 0.125, 0, window=(3, 4)), ptrs(14)) == 0
    assert bob(lib, S(1, 1, 0, 64, 0.125, 1, window=(0, -1)), ptrs(14)) == 0


def test_rejects_bad_sequence_offsets(lib):
    def shape(seq, nseq, N=128):
        return fbob.fbob_shape(1, 1, N, 64, 0.125, 0, -1, -1, seq, nseq)
    assert bob(lib, shape(None, 3), ptrs(14)) == 1               # count without offsets
    assert bob(lib, shape(BASE, 0), ptrs(14)) == 1               # offsets without a count
    assert bob(lib, shape(BASE + 2, 2), ptrs(14)) == 1           # misaligned offsets
    assert bob(lib, shape(BASE, (1 << 24) + 1), ptrs(14)) == 1   # more sequences than N allows
    assert bob(lib, shape(BASE, 2, N=0), ptrs(14)) == 0          # valid: empty problem, no call


def test_rejects_bad_kv_heads(lib):
    def shape(H, Hkv, N=128):
        return fbob.fbob_shape(1, H, N, 64, 0.125, 0, -1, -1, None, 0, Hkv)
    assert bob(lib, shape(4, 3), ptrs(14)) == 1       # not a divisor of H
    assert bob(lib, shape(4, -1), ptrs(14)) == 1
    assert bob(lib, shape(4, 2, N=0), ptrs(14)) == 0  # valid: empty problem, no call
    assert bob(lib, shape(4, 0, N=0), ptrs(14)) == 0  # 0 = no grouping


def test_rejects_bad_dropout_rates(lib):
    S = fbob.make_shape
    for p in (1.0, 1.5, -0.01, float("nan"), float("inf")):
        assert bob(lib, S(1, 1, 128, 64, 0.125, 0, dropout=(p, 3)), ptrs(14)) == 1, p
        assert lib.fbob_attn_fwd(ctypes.byref(S(1, 1, 128, 64, 0.125, 0, dropout=(p, 3))),
                                 *ptrs(5), None) == 1, p
    # valid rates (and any 64-bit seed) pass validation, then stop at the empty problem
    for p in (0.0, 0.001, 0.5, 0.999):
        assert bob(lib, S(1, 1, 0, 64, 0.125, 1, dropout=(p, (1 << 64) - 1)), ptrs(14)) == 0


def test_shape_struct_matches_the_header():
    """The ctypes mirror lists the C struct's fields in the header's order."""
    import re
    text = open(fbob.HEADER).read()
    body = re.search(r"typedef struct fbob_shape \{(.*?)\} fbob_shape;", text, re.S).group(1)
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    declared = re.findall(r"(\w+)\s*(?=[,;])", body)
    assert declared == [f[0] for f in fbob.fbob_shape._fields_]


def test_head_dim_32_passes_validation(lib):
    S = fbob.make_shape
    assert bob(lib, S(1, 1, 0, 32, 0.17, 1), ptrs(14)) == 0  # valid: empty problem, no call
    assert bob(lib, S(1, 1, 128, 32, 0.17, 1), ptrs(14, misalign=3)) == 1


def test_host_buffer_bob_validates_before_any_cuda_call(lib):
    S = fbob.make_shape
    shp = S(2, 4, 256, 64, 0.125, 1, kv_heads=2)
    host = ptrs(14)
    ws = ctypes.c_void_p(BASE + 20 * STRIDE)
    call = lib.fbob_attn_bob_host
    # (every call below fails validation or is empty: none reaches a CUDA call)
    # null host pointer, misaligned or null workspace, negative size, overlapping outputs
    bad = list(host)
    bad[3] = None
    assert call(ctypes.byref(shp), *bad, ws, 1 << 30, None) == 1
    assert call(ctypes.byref(shp), *host, ctypes.c_void_p(BASE + 20 * STRIDE + 16), 1 << 30,
                None) == 1
    assert call(ctypes.byref(shp), *host, None, 1 << 30, None) == 1
    assert call(ctypes.byref(shp), *host, ws, -1, None) == 1
    ov = list(host)
    ov[10] = ov[9]  # k_bar aliases q_bar
    assert call(ctypes.byref(shp), *ov, ws, 1 << 30, None) == 1
    # a workspace that cannot hold one key/value group of 2 query heads
    assert call(ctypes.byref(shp), *host, ws, 1024, None) == 1
    # empty problem: valid, no CUDA call
    assert call(ctypes.byref(S(0, 4, 256, 64, 0.125, 1)), *host, ws, 0, None) == 0
    assert lib.fbob_launch_count(b"bob_host") == 0


def test_host_workspace_size(lib):
    S = fbob.make_shape
    shp = S(2, 8, 1000, 128, 0.09, 1, kv_heads=2)   # groups of 4 query heads
    one = lib.fbob_attn_bob_host_workspace(ctypes.byref(shp), 1)
    assert one == lib.fbob_attn_bob_host_workspace(ctypes.byref(shp), 4)   # rounded up to a group
    nd = 1000 * 128 * 2
    # two slots of: 4 query-side + 2 output query-side + lse + row_stats, 4 + 2 key/value-side
    want = 2 * (6 * 4 * nd + 6 * 1 * nd + 4 * 1000 * 4 + 3 * 4 * 1000 * 4)
    assert want <= one <= want + 2 * 14 * 256
    assert lib.fbob_attn_bob_host_workspace(ctypes.byref(shp), 0) == -1
    assert lib.fbob_attn_bob_host_workspace(ctypes.byref(S(1, 1, 8, 48, 0.1, 0)), 1) == -1


def test_noalloc_host_bob_refuses_before_any_cuda_call(lib):
    S = fbob.make_shape
    call = lib.fbob_attn_bob_host_noalloc
    host = ptrs(14)
    # one key/value group of 4 heads at N = 16384, d = 128 needs ~193 MiB > 64 MiB
    assert call(ctypes.byref(S(1, 8, 16384, 128, 0.09, 1, kv_heads=2)), *host, None) == 6
    assert lib.fbob_status_string(6) == b"FBOB_ERR_SCRATCH_LIMIT"
    bad = list(host)
    bad[0] = None
    assert call(ctypes.byref(S(1, 1, 128, 64, 0.125, 0)), *bad, None) == 1
    assert call(ctypes.byref(S(0, 1, 128, 64, 0.125, 0)), *host, None) == 0  # empty: no call
    assert lib.fbob_launch_count(b"bob_host_noalloc") == 0
