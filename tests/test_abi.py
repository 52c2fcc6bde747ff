"""The C-ABI library loads on the CPU, exports every symbol include/bp.h
declares, its ctypes mirror matches the C structs, and argument checks that
run on the host reject bad calls without touching a GPU."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2111_11581_gb300 import bp, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "bp.h")


@pytest.fixture(scope="module")
def lib():
    build.build()
    return bp.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(bp_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_binding_exports():
    assert declared_functions() == sorted(bp.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", bp.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (bp_\w+)", out))
    for name in declared_functions():
        assert name in exported, name
        assert hasattr(lib, name)


def test_ctypes_structs_match_header(tmp_path):
    src = tmp_path / "sz.c"
    src.write_text('#include "bp.h"\n#include <stdio.h>\n#include <stddef.h>\n'
                   'int main(void){printf("%zu %zu %zu %zu %zu %zu\\n", sizeof(bp_layout),'
                   ' offsetof(bp_layout, K), offsetof(bp_layout, bk), sizeof(bp_packed),'
                   ' offsetof(bp_packed, rb_ptr), offsetof(bp_packed, dev_bytes)); return 0;}\n')
    exe = tmp_path / "sz"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)],
                   check=True)
    got = list(map(int, subprocess.run([str(exe)], capture_output=True, text=True,
                                       check=True).stdout.split()))
    want = [ctypes.sizeof(bp.Layout), bp.Layout.K.offset, bp.Layout.bk.offset,
            ctypes.sizeof(bp.Packed), bp.Packed.rb_ptr.offset, bp.Packed.dev_bytes.offset]
    assert got == want


def test_status_strings_and_version(lib):
    assert bp.status_string(bp.OK) == "ok"
    assert bp.status_string(bp.ERR_TIMEOUT) == "kernel wait timed out"
    assert bp.bp_version() >> 16 == 2 and bp.bp_version() & 0xffff >= 4


def test_workspace_size_is_host_only(lib):
    lay = bp.layout(bp.BLOCK_BASED, bp.BF16, 4096, 4096, 128, 32)
    n = bp.bp_workspace_size(lay)
    # fp64 score + keep byte per unit (RB * K units) plus small tables
    assert n >= 32 * 4096 * 9
    with pytest.raises(bp.BpError):
        bp.bp_workspace_size(bp.layout(bp.BLOCK_BASED, bp.BF16, 0, 16, 16, 16))


@pytest.mark.parametrize("bad", [
    dict(scheme=2), dict(dtype=7), dict(M=0), dict(K=0), dict(bm=0), dict(bk=0),
    dict(kh=3, kw=3, K=10),            # K not a multiple of kh*kw
])
def test_host_argument_checks(lib, bad):
    args = dict(scheme=0, dtype=1, M=64, K=64, bm=16, bk=16, kh=1, kw=1)
    args.update(bad)
    lay = bp.Layout(args["scheme"], args["dtype"], args["M"], args["K"], args["kh"], args["kw"],
                    args["bm"], args["bk"])
    assert bp.bp_prune(lay, 16, 2.0, 16, 256, 1 << 20, 0) == bp.ERR_INVALID_ARG


def test_rate_below_one_rejected_on_host(lib):
    lay = bp.layout(bp.BLOCK_BASED, bp.F16, 64, 64, 16, 16)
    assert bp.bp_prune(lay, 16, 0.5, 16, 256, 1 << 20, 0) == bp.ERR_INVALID_ARG
    assert bp.bp_prune(lay, 16, float("nan"), 16, 256, 1 << 20, 0) == bp.ERR_INVALID_ARG
    assert bp.bp_prune(lay, 16, 2.0, 16, 256, 16, 0) == bp.ERR_WORKSPACE


def test_noalloc_checks_on_host(lib):
    # rejected before any device call: a layout whose workspace exceeds the
    # library's 8 MiB scratch array, and an invalid layout
    big = bp.layout(bp.BLOCK_BASED, bp.BF16, 8192, 8192, 1, 1)
    assert bp.bp_workspace_size(big) > 8 << 20
    assert bp.bp_prune_noalloc(big, 16, 2.0, 16, 0) == bp.ERR_WORKSPACE
    bad = bp.Layout(0, 1, 64, 64, 1, 1, 0, 16)                        # bm = 0
    assert bp.bp_prune_noalloc(bad, 16, 2.0, 16, 0) == bp.ERR_INVALID_ARG


def test_gemm_argument_checks_on_host(lib):
    lay = bp.layout(bp.BLOCK_BASED, bp.F16, 64, 64, 16, 16)
    P = bp.Packed(lay, 4, 0, 0, 16, 16, 16, 256, 256 + 16384 + 640 + 4 * 64)   # kc_ptr, one chunk, qmap
    # ldx not a multiple of 8, misaligned X, N > ldx, null packed
    assert bp.bp_gemm(P, 256, 10, 10, None, 0, 256, 16, 0) == bp.ERR_INVALID_ARG
    assert bp.bp_gemm(P, 258, 8, 8, None, 0, 256, 8, 0) == bp.ERR_INVALID_ARG
    assert bp.bp_gemm(P, 256, 16, 8, None, 0, 256, 16, 0) == bp.ERR_INVALID_ARG
    assert bp.load().bp_gemm(None, 256, 8, 8, None, 0, 256, 8, None, 0, None) == bp.ERR_INVALID_ARG
    # a workspace must be 256-byte aligned and as large as bp_gemm_workspace_size says
    st, n = bp.bp_gemm_workspace_size(P, 8)
    assert st == bp.OK
    assert bp.bp_gemm(P, 256, 8, 8, None, 0, 256, 8, 256 + 16, 1 << 30) == bp.ERR_WORKSPACE
    if n:
        assert bp.bp_gemm(P, 256, 8, 8, None, 0, 256, 8, 1 << 20, n - 1) == bp.ERR_WORKSPACE
    # an image size that is not kc_ptr + whole (tile, record) chunks
    Pbad = bp.Packed(lay, 4, 0, 0, 16, 16, 16, 256, 256 + 16384)
    assert bp.bp_gemm(Pbad, 256, 8, 8, None, 0, 256, 8, 0) == bp.ERR_INVALID_ARG
    # more than 8192 slabs of 128 rows (M > 1,048,576) is beyond the device image
    M2 = (1 << 20) + 128
    lay2 = bp.layout(bp.BLOCK_BASED, bp.F16, M2, 64, 16, 16)
    P2 = bp.Packed(lay2, M2 // 16, 0, 0, 16, 16, 16, 256, 1 << 20)
    assert bp.bp_gemm(P2, 256, 8, 8, None, 0, 256, 8, 0) == bp.ERR_UNSUPPORTED


def test_conv_argument_checks_on_host(lib):
    lay = bp.layout(bp.BLOCK_PUNCHED, bp.F16, 16, 8 * 9, 8, 4, 3, 3)
    # kc_ptr, one chunk, qmap; then (256-byte aligned) the implicit convolution's
    # section, sized for all 9 K-groups (64 channels at each of 9 positions)
    head = 256 + 16384 + 640 + 4 * 72
    sec3 = 256 + 9 * (16384 + 320)
    P = bp.Packed(lay, 2, 0, 0, 16, 16, 16, 256, (head + 255) // 256 * 256 + sec3)
    # C*kh*kw != K, negative pad, zero stride
    ws = 1 << 16
    assert bp.bp_conv2d(P, 256, 2, 7, 8, 8, 1, 1, 1, 1, None, 0, 256, ws, 1 << 20, 0) == \
        bp.ERR_INVALID_ARG
    assert bp.bp_conv2d(P, 256, 2, 8, 8, 8, -1, 1, 1, 1, None, 0, 256, ws, 1 << 20, 0) == \
        bp.ERR_INVALID_ARG
    assert bp.bp_conv2d(P, 256, 2, 8, 8, 8, 1, 1, 0, 1, None, 0, 256, ws, 1 << 20, 0) == \
        bp.ERR_INVALID_ARG
    # (batches with at least 160 output tiles: launches that fill the SMs of a
    # GPU, if one is present, without splitting, so no partial tiles are added)
    # stride 1: the implicit convolution's workspace, the input in NHWC with the
    # channels padded to 8: 640 x 8 x 8 x 8 16-bit values (4 images per tile)
    assert bp.bp_conv2d_workspace_size(P, 640, 8, 8, 8, 1, 1, 1, 1) == \
        (bp.OK, 640 * 8 * 8 * 8 * 2)
    # stride 2 both ways: the input's four phases, each ceil(7/2) x ceil(7/2)
    # pixels of 8 channels (4 x 4 outputs: 16 images per tile)
    assert bp.bp_conv2d_workspace_size(P, 2560, 8, 7, 7, 1, 1, 2, 2) == \
        (bp.OK, 4 * 2560 * 4 * 4 * 8 * 2)
    # other strides: the im2col workspace, K x roundup8(Nb*Ho*Wo) 16-bit values
    assert bp.bp_conv2d_workspace_size(P, 4400, 8, 7, 5, 0, 0, 2, 1) == \
        (bp.OK, 72 * 39600 * 2)
    assert bp.bp_conv2d_workspace_size(P, 2, 7, 8, 8, 1, 1, 1, 1)[0] == bp.ERR_INVALID_ARG
    # too small, missing or misaligned workspace
    assert bp.bp_conv2d(P, 256, 2, 8, 8, 8, 1, 1, 1, 1, None, 0, 256, ws, 2 * 8 * 8 * 8 * 2 - 1,
                        0) == bp.ERR_WORKSPACE
    assert bp.bp_conv2d(P, 256, 3, 8, 7, 5, 0, 0, 2, 1, None, 0, 256, ws, 72 * 32 * 2 - 1, 0) \
        == bp.ERR_WORKSPACE
    assert bp.bp_conv2d(P, 256, 2, 8, 8, 8, 1, 1, 1, 1, None, 0, 256, None, 1 << 20, 0) == \
        bp.ERR_WORKSPACE
    assert bp.bp_conv2d(P, 256, 2, 8, 8, 8, 1, 1, 1, 1, None, 0, 256, ws + 8, 1 << 20, 0) == \
        bp.ERR_WORKSPACE


def test_penalty_argument_checks_on_host(lib):
    lay = bp.layout(bp.BLOCK_BASED, bp.BF16, 256, 512, 128, 32)
    assert bp.bp_penalty_units(lay) == (bp.OK, 2 * 512)
    play = bp.layout(bp.BLOCK_PUNCHED, bp.F16, 24, 5 * 9, 8, 2, 3, 3)
    assert bp.bp_penalty_units(play) == (bp.OK, 3 * 3 * 9)      # 3 filter blocks x 3 channel blocks
    # tiles of 128 rows x 64 columns (32 slices of 4 rows): 2 row-blocks x 8 tiles
    assert bp.bp_penalty_workspace_size(lay) == (bp.OK, 256 + 8 * 16)
    # one thread per unit: 81 units -> one block
    assert bp.bp_penalty_workspace_size(play) == (bp.OK, 256 + 8)
    a = 1 << 20
    # eps must be positive and finite, lambda finite, W / grad 16-B aligned
    for eps, lam in ((0.0, 1.0), (-1.0, 1.0), (float("inf"), 1.0), (1e-4, float("nan"))):
        assert bp.bp_reweighted_penalty(lay, 0, a, eps, lam, a, a, a, a, 1 << 16, 0) == \
            bp.ERR_INVALID_ARG
    assert bp.bp_reweighted_penalty(lay, 0, a + 8, 1e-4, 1.0, a, a, a, a, 1 << 16, 0) == \
        bp.ERR_INVALID_ARG
    assert bp.bp_reweighted_penalty(lay, 0, a, 1e-4, 1.0, a, a, a + 4, a, 1 << 16, 0) == \
        bp.ERR_INVALID_ARG
    # outside the fp32 range of the factors
    for eps, lam in ((2.0 ** -61, 1.0), (2.0 ** 61, 1.0), (1e-18, 1e3)):
        assert bp.bp_reweighted_penalty(lay, 0, a, eps, lam, a, a, a, a, 1 << 16, 0) == \
            bp.ERR_UNSUPPORTED
    # missing, misaligned or short workspace
    assert bp.bp_reweighted_penalty(lay, 0, a, 1e-4, 1.0, a, a, a, None, 1 << 16, 0) == \
        bp.ERR_WORKSPACE
    assert bp.bp_reweighted_penalty(lay, 0, a, 1e-4, 1.0, a, a, a, a + 16, 1 << 16, 0) == \
        bp.ERR_WORKSPACE
    assert bp.bp_reweighted_penalty(lay, 0, a, 1e-4, 1.0, a, a, a, a, 256 + 8 * 16 - 1, 0) == \
        bp.ERR_WORKSPACE
    # row groups (Eq. row): M x ceil(K / bk) segments; bk = 32 divides K: eight warps of
    # 256 weights per block (64 blocks); bk = 7: one thread per segment (37 blocks)
    assert bp.bp_penalty_units(lay, bp.GROUPS_ROWS) == (bp.OK, 256 * 16)
    assert bp.bp_penalty_workspace_size(lay, bp.GROUPS_ROWS) == (bp.OK, 256 + 8 * 64)
    lay7 = bp.layout(bp.BLOCK_BASED, bp.BF16, 128, 512, 128, 7)
    assert bp.bp_penalty_units(lay7, bp.GROUPS_ROWS) == (bp.OK, 128 * 74)
    assert bp.bp_penalty_workspace_size(lay7, bp.GROUPS_ROWS) == (bp.OK, 256 + 8 * 37)
    assert bp.bp_penalty_units(play, bp.GROUPS_ROWS)[0] == bp.ERR_INVALID_ARG
    assert bp.bp_penalty_units(lay, 2)[0] == bp.ERR_INVALID_ARG
    assert bp.bp_reweighted_penalty(play, bp.GROUPS_ROWS, a, 1e-4, 1.0, a, a, a, a, 1 << 16, 0) \
        == bp.ERR_INVALID_ARG
    # M*K >= 2^31 is outside the kernels' 32-bit indexing
    big = bp.layout(bp.BLOCK_BASED, bp.BF16, 1 << 16, 1 << 15, 128, 32)
    assert bp.bp_penalty_workspace_size(big)[0] == bp.ERR_UNSUPPORTED


def test_prune_rows_argument_checks_on_host(lib):
    lay = bp.layout(bp.BLOCK_BASED, bp.F16, 256, 64, 128, 8)
    # one workspace serves both: row units (256 x 8 = 2048) outnumber column units (2 x 64)
    n = bp.bp_workspace_size(lay)
    lay_cols_only = bp.layout(bp.BLOCK_BASED, bp.F16, 256, 64, 128, 128)
    assert n >= 2048 * 8 + 2048 and n > bp.bp_workspace_size(lay_cols_only)
    a = 1 << 20
    assert bp.bp_prune_rows(lay, a, 0.5, a, a, n, 0) == bp.ERR_INVALID_ARG
    assert bp.bp_prune_rows(lay, a, 2.0, a, a, n - 1, 0) == bp.ERR_WORKSPACE
    play = bp.layout(bp.BLOCK_PUNCHED, bp.F16, 16, 8 * 9, 8, 4, 3, 3)
    assert bp.bp_prune_rows(play, a, 2.0, a, a, 1 << 20, 0) == bp.ERR_INVALID_ARG


def test_prune_pattern_argument_checks_on_host(lib):
    lay = bp.layout(bp.BLOCK_PUNCHED, bp.F16, 64, 32 * 9, 8, 4, 3, 3)
    n = bp.bp_workspace_size(lay)
    a = 1 << 20
    pats = list(bp.DEFAULT_PATTERNS)
    assert bp.bp_prune_pattern(lay, a, 2.0, pats, a, a, n, 0) == bp.ERR_INVALID_ARG      # rate < 9/4
    assert bp.bp_prune_pattern(lay, a, 4.0, [0b111], a, a, n, 0) == bp.ERR_INVALID_ARG   # 3 entries
    assert bp.bp_prune_pattern(lay, a, 4.0, [1 << 9 | 0b111], a, a, n, 0) == bp.ERR_INVALID_ARG
    assert bp.bp_prune_pattern(lay, a, 4.0, pats * 3, a, a, n, 0) == bp.ERR_INVALID_ARG  # 24 > 16
    assert bp.bp_prune_pattern(lay, a, 4.0, pats, a, a, n - 1, 0) == bp.ERR_WORKSPACE
    for other in (bp.layout(bp.BLOCK_PUNCHED, bp.F16, 64, 32 * 25, 8, 4, 5, 5),
                  bp.layout(bp.BLOCK_BASED, bp.F16, 64, 288, 8, 4)):
        assert bp.bp_prune_pattern(other, a, 4.0, pats, a, a, 1 << 22, 0) == bp.ERR_INVALID_ARG
    # the workspace covers one unit per kernel (64 x 32) plus its pattern byte
    assert n >= 64 * 32 * (8 + 1 + 1)
