"""The C-ABI library without a GPU: it loads, exports every function that
include/bigcn.h declares, and its host-side argument checks return the
documented status before any CUDA call is made (fake, never-dereferenced
pointers are enough to reach them)."""
import ctypes
import os
import re

import pytest

from paper_2010_07565_gb300 import build as lib_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "bigcn.h")

OK, INVALID, MISALIGNED = 0, 1, 2
P = 1 << 32          # a fake, 256-byte-aligned device address (never dereferenced)


@pytest.fixture(scope="module")
def lib():
    from paper_2010_07565_gb300 import binding
    lib_build.build()
    return binding.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(bigcn_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_five_steps_and_helpers():
    names = declared_functions()
    for n in ["bigcn_pack_rows", "bigcn_pack_weights", "bigcn_xnor_gemm", "bigcn_spmm_norm",
              "bigcn_layer_forward", "bigcn_layer_workspace_bytes", "bigcn_words",
              "bigcn_status_string"]:
        assert n in names


def test_library_exports_every_declared_function(lib):
    for name in declared_functions():
        assert hasattr(lib, name), f"{name} is declared in bigcn.h but not exported"


def test_binding_covers_every_declared_function():
    from paper_2010_07565_gb300 import binding
    for name in declared_functions():
        assert name in binding.SIGNATURES


def test_words_and_status_strings(lib):
    assert [lib.bigcn_words(k) for k in (-3, 0, 1, 63, 64, 65, 128, 8192)] == \
        [0, 0, 1, 1, 1, 2, 2, 128]
    assert lib.bigcn_status_string(0) == b"BIGCN_OK"
    assert lib.bigcn_status_string(2) == b"BIGCN_ERR_MISALIGNED"
    assert lib.bigcn_status_string(99) == b"BIGCN_ERR_UNKNOWN"


def test_workspace_bytes(lib):
    assert lib.bigcn_layer_workspace_bytes(0, 0, 5) == 0
    assert lib.bigcn_layer_workspace_bytes(-1, 10, 5) == 0
    # K <= 2048, F <= 128: Z kept factored as fp16 dots (rows padded to 16) plus
    # a row scale
    n = lib.bigcn_layer_workspace_bytes(1000, 130, 62)
    need = 1000 * 3 * 8 + 1000 * 4 + 62 * 3 * 8 + 62 * 4 + 1000 * 64 * 2 + 1000 * 4
    assert need <= n <= need + 7 * 256 and n % 256 == 0
    assert lib.bigcn_layer_workspace_bytes(2000, 130, 62) > n
    # K > 2048: uint16 dots (rows padded to 8); K >= 4096: also the weight signs
    # as the tensor-core product's FP8 tiles (one 64-column tile x 33 k-blocks
    # of 128 bytes a row)
    n = lib.bigcn_layer_workspace_bytes(1000, 4100, 62)
    need = (1000 * 65 * 8 + 1000 * 4 + 62 * 65 * 8 + 62 * 4 + 1000 * 64 * 2 + 1000 * 4 +
            1 * 33 * 64 * 128)
    assert need <= n <= need + 7 * 256 and n % 256 == 0
    # larger K: fp32 Z
    n = lib.bigcn_layer_workspace_bytes(100, 40000, 5)
    need = 100 * 625 * 8 + 100 * 4 + 5 * 625 * 8 + 5 * 4 + 100 * 5 * 4
    assert need <= n <= need + 7 * 256 and n % 256 == 0


def test_pack_rows_argument_checks(lib):
    f = lib.bigcn_pack_rows
    assert f(P, 0, 10, 10, None, None, P + 4096, 1, P + 8192, None) == OK      # N = 0
    assert f(P, 4, 0, 10, None, None, P + 4096, 1, P + 8192, None) == INVALID  # K = 0
    assert f(P, 4, 10, 9, None, None, P + 4096, 1, P + 8192, None) == INVALID  # ldx < K
    assert f(P, 4, 65, 65, None, None, P + 4096, 1, P + 8192, None) == INVALID  # words
    assert f(None, 4, 10, 10, None, None, P + 4096, 1, P + 8192, None) == INVALID
    assert f(P, 4, 10, 10, P + 512, None, P + 4096, 1, P + 8192, None) == INVALID  # one NULL
    assert f(P + 2, 4, 10, 10, None, None, P + 4096, 1, P + 8192, None) == MISALIGNED
    assert f(P, 4, 10, 10, None, None, P + 4100, 1, P + 8192, None) == MISALIGNED
    assert f(P, 4, 10, 10, None, None, P + 8, 1, P + 8192, None) == INVALID    # bits overlap X
    assert f(P, 1 << 40, 10, 1 << 30, None, None, P + 4096, 1, P + 8192, None) == INVALID


def test_pack_weights_argument_checks(lib):
    f = lib.bigcn_pack_weights
    assert f(P, 10, 0, 1, P + 4096, 1, P + 8192, None) == INVALID
    assert f(P, 10, 4, 3, P + 4096, 1, P + 8192, None) == INVALID               # ldw < F
    assert f(P, 10, 4, 4, None, 1, P + 8192, None) == INVALID
    assert f(P, 10, 4, 4, P + 4, 1, P + 8192, None) == MISALIGNED
    assert f(P, 10, 4, 4, P + 16, 1, P + 8192, None) == INVALID                 # overlap


def test_xnor_gemm_argument_checks(lib):
    f = lib.bigcn_xnor_gemm
    a, al, b, be, z = P, P + 65536, P + 2 * 65536, P + 3 * 65536, P + 4 * 65536
    assert f(a, al, 0, b, be, 4, 10, 1, z, 4, None, None) == OK
    assert f(a, al, 8, b, be, 0, 10, 1, z, 4, None, None) == INVALID
    assert f(a, al, 8, b, be, 4, 65, 1, z, 4, None, None) == INVALID             # words
    assert f(a, al, 8, b, be, 4, 10, 1, z, 3, None, None) == INVALID             # ldz < F
    assert f(a + 4, al, 8, b, be, 4, 10, 1, z, 4, None, None) == MISALIGNED
    assert f(a, al, 8, b, be, 4, 10, 1, z, 4, z + 2, None) == MISALIGNED         # dots
    assert f(a, al, 8, b, be, 4, 10, 1, a, 4, None, None) == INVALID             # Z aliases A
    assert f(a, al, 8, b, be, 4, 10, 1, z, 4, z, None) == INVALID                # dots alias Z


def test_spmm_argument_checks(lib):
    f = lib.bigcn_spmm_norm
    rp, ci, z, h = P, P + 65536, P + 2 * 65536, P + 3 * 65536
    assert f(rp, ci, 0, 0, z, 4, 4, h, 4, None) == OK
    assert f(rp, ci, 1 << 31, 10, z, 4, 4, h, 4, None) == INVALID                # N > INT32_MAX
    assert f(rp, ci, 8, -1, z, 4, 4, h, 4, None) == INVALID
    assert f(rp, None, 8, 5, z, 4, 4, h, 4, None) == INVALID                     # colidx NULL
    assert f(rp + 4, ci, 8, 5, z, 4, 4, h, 4, None) == MISALIGNED
    assert f(rp, ci, 8, 5, z, 4, 4, z + 16, 4, None) == INVALID                  # H overlaps Z
    assert f(rp, ci, 8, 5, z, 4, 4, h, 3, None) == INVALID                       # ldh < F


def test_layer_forward_argument_checks(lib):
    f = lib.bigcn_layer_forward
    X, W, rp, ci, ws, H = (P + q * (1 << 24) for q in range(6))
    need = lib.bigcn_layer_workspace_bytes(100, 70, 8)
    args = lambda **kw: [kw.get("X", X), kw.get("N", 100), 70, 70, None, None, W, 8, 8, rp, ci,
                         300, kw.get("ws", ws), kw.get("wsb", need), kw.get("H", H), 8, None]
    assert f(*args(N=0)) == OK
    assert f(*args(wsb=need - 1)) == INVALID
    assert f(*args(ws=ws + 128)) == MISALIGNED                                   # 256-B alignment
    assert f(*args(ws=X)) == INVALID                                              # overlaps X
    assert f(*args(H=ws + 256)) == INVALID                                        # H in workspace
    assert f(*args(H=X)) == INVALID


def test_forward_2layer_aggregation_query(lib):
    """The 2-layer forward aggregates on the tensor cores exactly when layer 1's
    dots fit fp16 (K <= 2048), Fh <= 128 and Fo <= 64; the query needs no GPU."""
    from paper_2010_07565_gb300 import binding as B
    assert B.bigcn_forward_2layer_aggregation(602, 128, 41) == 1      # Reddit-shaped
    assert B.bigcn_forward_2layer_aggregation(1433, 64, 7) == 1       # Cora-shaped
    assert B.bigcn_forward_2layer_aggregation(2048, 30, 64) == 1
    assert B.bigcn_forward_2layer_aggregation(3703, 64, 6) == 0       # Citeseer-shaped
    assert B.bigcn_forward_2layer_aggregation(2049, 64, 7) == 0
    assert B.bigcn_forward_2layer_aggregation(500, 129, 7) == 0
    assert B.bigcn_forward_2layer_aggregation(500, 64, 65) == 0
    with pytest.raises(B.BigcnError):
        B.bigcn_forward_2layer_aggregation(0, 64, 7)
