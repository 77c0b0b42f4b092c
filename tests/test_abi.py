"""The C-ABI library on the CPU: it loads, exports every declared symbol,
rejects bad arguments before touching CUDA, and plans the work decomposition
consistently.  No compute call is made here (no GPU in this process)."""
import ctypes
import os
import re

import pytest

import paper_2512_22147_gb300 as dm
from paper_2512_22147_gb300 import _binding as B

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                      "include", "dualmv.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(dualmv_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_entry_points():
    names = declared_functions()
    for n in ("dualmv_f32", "dualmv_f64", "dualmv_i32", "dualmv_f32_strided_batched",
              "dualmv_f64_strided_batched", "dualmv_i32_strided_batched",
              "dualmv_status_string", "dualmv_device_fault", "dualmv_plan"):
        assert n in names


@pytest.mark.parametrize("name", declared_functions())
def test_library_exports_every_declared_symbol(name):
    lib = ctypes.CDLL(dm.LIBRARY_PATH)
    assert hasattr(lib, name), name
    assert name in B.EXPORTED


def test_library_is_in_tree_and_sm103a():
    assert os.path.dirname(dm.LIBRARY_PATH).endswith("paper_2512_22147_gb300")
    from paper_2512_22147_gb300 import build
    assert "arch=compute_103a,code=sm_103a" in build.NVCC_FLAGS


def test_status_strings():
    assert dm.dualmv_status_string(0) == "success"
    assert "invalid" in dm.dualmv_status_string(1)
    assert "allocation" in dm.dualmv_status_string(2)
    assert dm.dualmv_status_string(99) == "unknown status"


def test_set_path_round_trip():
    old = dm.dualmv_set_path(dm.DUALMV_PATH_DIRECT)
    assert dm.dualmv_set_path(old) == dm.DUALMV_PATH_DIRECT
    with pytest.raises(ValueError):
        dm.dualmv_set_path(7)


FAKE = 0x10000  # never dereferenced: every call below fails validation first


@pytest.mark.parametrize("args", [
    (-1, 4, FAKE, 4, FAKE, FAKE, FAKE, FAKE),    # M < 0
    (4, -1, FAKE, 4, FAKE, FAKE, FAKE, FAKE),    # N < 0
    (4, 8, FAKE, 7, FAKE, FAKE, FAKE, FAKE),     # lda < N
    (4, 0, FAKE, 0, FAKE, FAKE, FAKE, FAKE),     # lda < 1
    (4, 8, None, 8, FAKE, FAKE, FAKE, FAKE),     # A missing
    (4, 8, FAKE, 8, None, FAKE, FAKE, FAKE),     # p missing
    (4, 8, FAKE, 8, FAKE, None, FAKE, FAKE),     # r missing
    (4, 8, FAKE, 8, FAKE, FAKE, None, FAKE),     # q missing
    (4, 8, FAKE, 8, FAKE, FAKE, FAKE, None),     # s missing
    (4, 0, FAKE, 1, FAKE, FAKE, None, FAKE),     # q missing although N == 0
])
@pytest.mark.parametrize("tag", ["f32", "f64", "i32"])
def test_invalid_arguments_are_rejected(tag, args):
    fn = getattr(dm, f"dualmv_{tag}")
    assert fn(*args, None) == dm.DUALMV_ERR_INVALID_VALUE


@pytest.mark.parametrize("tag", ["f32", "f64", "i32"])
def test_invalid_batched_arguments(tag):
    fn = getattr(dm, f"dualmv_{tag}_strided_batched")
    ok = dict(M=4, N=8, A=FAKE, lda=8, sA=32, p=FAKE, sP=8, r=FAKE, sR=4, q=FAKE, sQ=4,
              s=FAKE, sS=8, batch=3)

    def call(**kw):
        a = dict(ok, **kw)
        return fn(a["M"], a["N"], a["A"], a["lda"], a["sA"], a["p"], a["sP"], a["r"],
                  a["sR"], a["q"], a["sQ"], a["s"], a["sS"], a["batch"], None)

    assert call(batch=-1) == dm.DUALMV_ERR_INVALID_VALUE
    assert call(sQ=3) == dm.DUALMV_ERR_INVALID_VALUE      # outputs overlap
    assert call(sS=7) == dm.DUALMV_ERR_INVALID_VALUE
    assert call(sA=-1) == dm.DUALMV_ERR_INVALID_VALUE
    assert call(sP=-8) == dm.DUALMV_ERR_INVALID_VALUE
    assert call(batch=0) == dm.DUALMV_SUCCESS              # nothing to do
    assert call(batch=0, M=-1) == dm.DUALMV_ERR_INVALID_VALUE


def test_fault_injection_alloc(monkeypatch):
    """An injected workspace-allocation failure is reported before any CUDA
    call, with nothing enqueued."""
    monkeypatch.setenv("DUALMV_FAULT_INJECT", "alloc")
    rc = dm.dualmv_f32(4, 8, FAKE, 8, FAKE, FAKE, FAKE, FAKE, None)
    assert rc == dm.DUALMV_ERR_ALLOC


# ------------------------------------------------------------- planner ----

def _ref_first(c, T, G):
    return (c * T) // G


@pytest.mark.parametrize("M,N,batch,eb,ab,sms", [
    (1024, 1024, 1, 4, 4, 152),
    (16384, 16384, 1, 4, 4, 152),
    (65536, 4096, 1, 8, 8, 152),
    (4001, 100003, 1, 4, 8, 152),
    (2048, 2048, 256, 4, 4, 152),
    (1, 1, 1, 4, 4, 152),
    (33, 257, 3, 8, 8, 7),
    (100, 5000, 2, 4, 8, 1),
])
def test_plan_covers_every_tile_once(M, N, batch, eb, ab, sms):
    pl = dm.dualmv_plan(M, N, batch, eb, ab, sms)
    # 4-byte types: 8 warps x 4 rows; fp64: 12 self-loading warps x 4 rows
    # (FP32-pipe kernel); all on 256-column bands
    rows, width = (48 if eb == 8 else 32, 256)
    assert pl.band_cols == width and pl.tile_rows == rows
    assert pl.bands == -(-N // width) and pl.stripes == -(-M // rows)
    assert pl.tiles == batch * pl.bands * pl.stripes
    assert pl.grid == min(pl.tiles, sms)
    T, G, S = pl.tiles, pl.grid, pl.stripes
    # Contiguous ranges partition [0, T) and differ in size by at most one.
    sizes = [_ref_first(c + 1, T, G) - _ref_first(c, T, G) for c in range(G)]
    assert sum(sizes) == T and max(sizes) - min(sizes) <= 1 and min(sizes) >= 1
    nseg = [(_ref_first(c + 1, T, G) - 1) // S - _ref_first(c, T, G) // S + 1
            for c in range(G)]
    assert pl.max_segments == max(nseg)
    q_ws = batch * pl.bands * M * ab if pl.bands > 1 else 0
    s_ws = G * pl.max_segments * width * ab
    if eb == 4 and ab == 8:          # int32: atomic exact sums, no workspace
        assert pl.workspace_bytes == 0
    else:
        assert pl.workspace_bytes == -(-q_ws // 256) * 256 + s_ws
    assert pl.smem_bytes <= 227 * 1024 and pl.threads == (288 if eb == 4 else 384)


def test_plan_rejects_bad_shapes():
    for args in ((0, 5, 1, 4, 4, 152), (5, 5, 1, 2, 4, 152), (5, 5, 1, 8, 4, 152),
                 (5, 5, 0, 4, 4, 152), (5, 5, 1, 4, 4, 0)):
        with pytest.raises(dm.DualmvError):
            dm.dualmv_plan(*args)
