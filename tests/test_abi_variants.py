"""Host-side logic of the C-ABI's variant entry points without a GPU:
workspace sizes and the argument checks of the ablation products and
layers, the inductive layers, sub-row bucketing, the layer backward and
the weighted-adjacency calls, which return their documented status before any CUDA call (fake,
never-dereferenced pointers are enough to reach them)."""
import pytest

from paper_2010_07565_gb300 import build as lib_build

OK, INVALID, MISALIGNED = 0, 1, 2
P = 1 << 32          # a fake, 256-byte-aligned device address (never dereferenced)
BOTH, WEIGHTS, FEATURES = 0, 1, 2
GCN, MEAN, SAGE = 0, 1, 2


@pytest.fixture(scope="module")
def lib():
    from paper_2010_07565_gb300 import binding
    lib_build.build()
    return binding.lib()


def ptrs(n, step=1 << 24):
    return [P + q * step for q in range(n)]


# ---------------------------------------------------------------- ablation --
def test_ablation_workspace_bytes(lib):
    f = lib.bigcn_layer_ablation_workspace_bytes
    assert f(BOTH, 1000, 130, 62) == lib.bigcn_layer_workspace_bytes(1000, 130, 62)
    assert f(7, 1000, 130, 62) == 0 and f(WEIGHTS, -1, 130, 62) == 0
    assert f(WEIGHTS, 10, 0, 4) == 0 and f(FEATURES, 10, 4, 0) == 0
    # weights binarized: W's packed columns + beta + Z (N x F fp32)
    n = f(WEIGHTS, 1000, 130, 62)
    need = 62 * 3 * 8 + 62 * 4 + 1000 * 62 * 4
    assert need <= n <= need + 4 * 256 and n % 256 == 0
    # features binarized: packed rows + alpha + W's three bf16 parts + Z
    n = f(FEATURES, 1000, 130, 62)
    need = 1000 * 3 * 8 + 1000 * 4 + 3 * 62 * 192 * 2 + 1000 * 62 * 4
    assert need <= n <= need + 4 * 256 and n % 256 == 0
    assert lib.bigcn_binary_real_gemm_workspace_bytes(130, 62) >= 3 * 62 * 192 * 2
    assert lib.bigcn_binary_real_gemm_workspace_bytes(0, 62) == 0


def test_real_binary_gemm_argument_checks(lib):
    f = lib.bigcn_real_binary_gemm
    X, bb, be, Z = ptrs(4)
    ok = lambda **kw: [kw.get("X", X), kw.get("N", 100), 70, kw.get("ldx", 70),
                       kw.get("s", None), kw.get("t", None), kw.get("bb", bb), be, 8,
                       kw.get("words", 2), kw.get("Z", Z), kw.get("ldz", 8), None]
    assert f(*ok(N=0)) == OK
    assert f(*ok(words=1)) == INVALID                            # words != ceil(K / 64)
    assert f(*ok(ldx=69)) == INVALID
    assert f(*ok(ldz=7)) == INVALID
    assert f(*ok(s=P + 5 * (1 << 24))) == INVALID                  # scale without shift
    assert f(*ok(X=X + 2)) == MISALIGNED
    assert f(*ok(bb=bb + 4)) == MISALIGNED
    assert f(*ok(Z=X + 256)) == INVALID                           # Z overlaps X


def test_binary_real_gemm_argument_checks(lib):
    f = lib.bigcn_binary_real_gemm
    A, al, W, ws, Z = ptrs(5)
    need = lib.bigcn_binary_real_gemm_workspace_bytes(70, 8)
    ok = lambda **kw: [A, al, kw.get("N", 100), 70, kw.get("words", 2), W, 8, kw.get("ldw", 8),
                       kw.get("ws", ws), kw.get("wsb", need), kw.get("Z", Z), 8, None]
    assert f(*ok(N=0)) == OK
    assert f(*ok(words=3)) == INVALID
    assert f(*ok(ldw=7)) == INVALID
    assert f(*ok(wsb=need - 1)) == INVALID
    assert f(*ok(ws=ws + 128)) == MISALIGNED
    assert f(*ok(ws=W)) == INVALID                                # workspace overlaps W
    assert f(*ok(Z=ws)) == INVALID                                # Z overlaps the workspace


def test_layer_ablation_argument_checks(lib):
    f = lib.bigcn_layer_forward_ablation
    X, W, rp, ci, ws, H = ptrs(6)
    for mode in (WEIGHTS, FEATURES):
        need = lib.bigcn_layer_ablation_workspace_bytes(mode, 100, 70, 8)
        args = lambda **kw: [kw.get("mode", mode), X, kw.get("N", 100), 70, 70, None, None, W, 8,
                             8, rp, ci, 300, kw.get("ws", ws), kw.get("wsb", need),
                             kw.get("H", H), 8, None]
        assert f(*args(N=0)) == OK
        assert f(*args(mode=9)) == INVALID
        assert f(*args(wsb=need - 1)) == INVALID
        assert f(*args(ws=ws + 128)) == MISALIGNED
        assert f(*args(H=X)) == INVALID


# --------------------------------------------------------------- inductive --
def test_inductive_workspace_bytes(lib):
    f = lib.bigcn_inductive_layer_workspace_bytes
    assert f(GCN, 1000, 130, 62) == lib.bigcn_layer_workspace_bytes(1000, 130, 62)
    assert f(5, 1000, 130, 62) == 0 and f(MEAN, 10, 0, 4) == 0
    mean, sage = f(MEAN, 1000, 130, 62), f(SAGE, 1000, 130, 62)
    # GraphSAGE: a product over 2 x 64 columns (each half padded to 8) instead of 62
    assert sage > mean and mean % 256 == 0 and sage % 256 == 0
    need = 1000 * 3 * 8 + 1000 * 4 + 128 * 3 * 8 + 128 * 4 + 1000 * 128 * 2 + 1000 * 4
    assert need <= sage <= need + 6 * 256
    # K past 32767: the products are fp32
    assert f(SAGE, 100, 40000, 8) >= 100 * 16 * 4


def test_inductive_argument_checks(lib):
    f = lib.bigcn_inductive_layer_forward
    X, W, Wn, rp, ci, ws, H = ptrs(7)
    need = lib.bigcn_inductive_layer_workspace_bytes(SAGE, 100, 70, 8)
    args = lambda **kw: [kw.get("agg", SAGE), X, kw.get("N", 100), 70, 70, None, None, W, 8, 8,
                         kw.get("Wn", Wn), kw.get("ldwn", 8), rp, ci, 300, kw.get("ws", ws),
                         kw.get("wsb", need), kw.get("H", H), 8, None]
    assert f(*args(N=0)) == OK
    assert f(*args(agg=7)) == INVALID
    assert f(*args(Wn=None)) == INVALID                            # GraphSAGE needs W_neigh
    assert f(*args(ldwn=7)) == INVALID
    assert f(*args(wsb=need - 1)) == INVALID
    assert f(*args(Wn=Wn + 2)) == MISALIGNED
    assert f(*args(ws=Wn)) == INVALID                              # workspace overlaps W_neigh
    # The mean aggregator ignores W_neigh.
    mneed = lib.bigcn_inductive_layer_workspace_bytes(MEAN, 100, 70, 8)
    assert f(*args(agg=MEAN, Wn=None, ldwn=0, wsb=mneed, N=0)) == OK


# ---------------------------------------------------------------- buckets --
def test_bucketed_workspace_bytes(lib):
    f = lib.bigcn_layer_bucketed_workspace_bytes
    assert f(100, 130, 8, 96) == 0 and f(100, 130, 8, 0) == 0 and f(100, 130, 8, -64) == 0
    n64, n128 = f(1000, 1433, 64, 64), f(1000, 1433, 64, 128)
    assert n64 > n128 > 0 and n64 % 256 == 0
    need = 1000 * 23 * 8 + 1000 * 23 * 4 + 64 * 23 * 8 + 64 * 23 * 4 + 1000 * 64 * 4
    assert need <= n64 <= need + 5 * 256
    assert f(10, 64 * 65536, 4, 64) == 0                           # more than 65535 buckets


def test_bucketed_argument_checks(lib):
    X, bits, al = ptrs(3)
    f = lib.bigcn_pack_rows_bucketed
    assert f(X, 0, 100, 100, None, None, 64, bits, 2, al, None) == OK
    for B in (0, 32, 100, -64):
        assert f(X, 4, 100, 100, None, None, B, bits, 2, al, None) == INVALID
    assert f(X, 4, 100, 100, None, None, 64, bits, 1, al, None) == INVALID  # words
    assert f(X + 2, 4, 100, 100, None, None, 64, bits, 2, al, None) == MISALIGNED
    g = lib.bigcn_xnor_gemm_bucketed
    A, a, Bb, b, Z = ptrs(5)
    assert g(A, a, 0, Bb, b, 4, 100, 2, 64, Z, 4, None) == OK
    assert g(A, a, 8, Bb, b, 4, 100, 3, 64, Z, 4, None) == INVALID      # words != ceil(K / 64)
    assert g(A, a, 8, Bb, b, 4, 100, 2, 96, Z, 4, None) == INVALID      # B not a multiple of 64
    assert g(A, a, 8, Bb, b, 4, 100, 2, 64, A, 4, None) == INVALID      # Z overlaps A


# ---------------------------------------------------------------- backward --
def test_backward_workspace_and_argument_checks(lib):
    ws_bytes = lib.bigcn_layer_backward_workspace_bytes
    assert ws_bytes(0, 0, 4) == 0 and ws_bytes(-1, 10, 4) == 0
    n = ws_bytes(1000, 130, 16)
    assert n >= 1000 * 3 * 8 + 1000 * 4 + 1000 * 16 * 4 + 130 * 16 * 4 and n % 256 == 0
    f = lib.bigcn_layer_backward
    X, W, rp, ci, dH, dX, dW, ws = ptrs(8)
    args = lambda **kw: [X, kw.get("N", 100), 70, 70, None, None, W, 8, 8, rp, ci, 300,
                         kw.get("dH", dH), 8, kw.get("dX", dX), 70, kw.get("dW", dW), 8, ws,
                         kw.get("wsb", ws_bytes(100, 70, 8)), None]
    assert f(*args(wsb=ws_bytes(100, 70, 8) - 1)) == INVALID
    assert f(*args(dW=None)) == INVALID
    assert f(*args(dW=dH)) == INVALID                              # dW overlaps dH
    assert f(*args(dX=dW)) == INVALID                              # dX overlaps dW
    assert f(*args(dX=dX + 2)) == MISALIGNED


# ------------------------------------------------------ weighted adjacency --
def test_weighted_workspace_bytes(lib):
    f = lib.bigcn_weighted_layer_workspace_bytes
    assert f(0, 0, 5) == 0 and f(-1, 10, 5) == 0
    # uint16 dots (rows padded to 8) + row scale, then dinv and s (N each)
    n = f(1000, 130, 62)
    need = (1000 * 3 * 8 + 1000 * 4 + 62 * 3 * 8 + 62 * 4 + 1000 * 64 * 2 + 1000 * 4 +
            2 * 1000 * 4)
    assert need <= n <= need + 9 * 256 and n % 256 == 0
    n = f(100, 40000, 5)                        # fp32 Z
    need = 100 * 625 * 8 + 100 * 4 + 5 * 625 * 8 + 5 * 4 + 100 * 5 * 4 + 2 * 100 * 4
    assert need <= n <= need + 9 * 256 and n % 256 == 0


def test_weighted_argument_checks(lib):
    d = lib.bigcn_weighted_dinv
    rp, v, dv = ptrs(3)
    assert d(rp, v, 0, 0, dv, None) == OK
    assert d(rp, None, 8, 5, dv, None) == INVALID       # values NULL with entries
    assert d(rp, v, -1, 5, dv, None) == INVALID
    assert d(rp, v, 8, -1, dv, None) == INVALID
    assert d(rp + 4, v, 8, 5, dv, None) == MISALIGNED
    assert d(rp, v + 2, 8, 5, dv, None) == MISALIGNED
    assert d(rp, v, 8, 5, v + 8, None) == INVALID       # dinv overlaps values
    s = lib.bigcn_spmm_norm_weighted
    rp, ci, v, dv, z, h = ptrs(6)
    assert s(rp, ci, v, dv, 0, 0, z, 4, 4, h, 4, None) == OK
    assert s(rp, ci, None, dv, 8, 5, z, 4, 4, h, 4, None) == INVALID        # values NULL
    assert s(rp, ci, v, None, 8, 5, z, 4, 4, h, 4, None) == INVALID         # dinv NULL
    assert s(rp, ci, v + 2, dv, 8, 5, z, 4, 4, h, 4, None) == MISALIGNED
    assert s(rp, ci, v, dv, 8, 5, z, 4, 4, v + 4, 4, None) == INVALID       # H overlaps values
    assert s(rp, ci, v, dv, 8, 5, z, 4, 4, dv, 4, None) == INVALID          # H overlaps dinv
    assert s(rp, ci, v, dv, 8, 5, z, 4, 4, h, 3, None) == INVALID           # ldh < F
    f = lib.bigcn_weighted_layer_forward
    X, W, rp, ci, v, ws, H = ptrs(7)
    need = lib.bigcn_weighted_layer_workspace_bytes(100, 70, 8)
    args = lambda **kw: [X, kw.get("N", 100), 70, 70, None, None, W, 8, 8, rp, ci,
                         kw.get("v", v), 300, kw.get("ws", ws), kw.get("wsb", need),
                         kw.get("H", H), 8, None]
    assert f(*args(N=0)) == OK
    assert f(*args(v=None)) == INVALID
    assert f(*args(v=v + 2)) == MISALIGNED
    assert f(*args(wsb=need - 1)) == INVALID
    assert f(*args(ws=ws + 128)) == MISALIGNED
    assert f(*args(ws=v)) == INVALID                    # workspace overlaps values
    assert f(*args(H=v)) == INVALID                     # H overlaps values
