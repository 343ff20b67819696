"""CPU-side checks of the C ABI: the library builds for sm_103a, loads without a
GPU, exports every entry point include/sdd.h declares, the ctypes mirror of
sdd_block_args matches the C layout, and host-side argument validation rejects
bad calls before touching the GPU."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sdd.h")


def _declared_functions():
    src = open(HEADER).read()
    return sorted(set(re.findall(r"^SDD_API\s+[^;(]*?\b(sdd_\w+)\s*\(", src, flags=re.M)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_14787_gb300 import build as b
    path = b.build()
    from paper_2608_14787_gb300 import binding
    return binding.load(path)


def test_header_declares_the_boundary():
    names = _declared_functions()
    for want in ("sdd_confidence", "sdd_schedule_prefix", "sdd_verify_strict", "sdd_verify_lenient",
                 "sdd_verify_topk", "sdd_block", "sdd_workspace_size"):
        assert want in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared_functions():
        assert hasattr(lib, name), name


def test_library_exports_nothing_else(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", lib._name], capture_output=True, text=True).stdout
    exported = sorted({line.split()[-1] for line in out.splitlines() if " T " in line})
    assert exported == _declared_functions()


def test_block_args_layout_matches_c(tmp_path):
    from paper_2608_14787_gb300.binding import BlockArgs
    fields = [f for f, _ in BlockArgs._fields_]
    prog = ["#include <stdio.h>", "#include <stddef.h>", f'#include "{HEADER}"', "int main(void) {",
            'printf("%zu\\n", sizeof(sdd_block_args));']
    for f in fields:
        prog.append(f'printf("%zu\\n", offsetof(sdd_block_args, {f}));')
    prog.append("return 0; }")
    c = tmp_path / "layout.c"
    c.write_text("\n".join(prog))
    exe = tmp_path / "layout"
    subprocess.check_call(["gcc", "-std=c11", "-o", str(exe), str(c)])
    vals = [int(x) for x in subprocess.check_output([str(exe)]).split()]
    assert vals[0] == ctypes.sizeof(BlockArgs)
    for f, off in zip(fields, vals[1:]):
        assert getattr(BlockArgs, f).offset == off, f


def test_version_and_error_string(lib):
    assert lib.sdd_version() >= 100
    assert isinstance(lib.sdd_last_error(), bytes)


def test_invalid_arguments_rejected_on_host(lib):
    from paper_2608_14787_gb300.binding import _f64_array
    VP = ctypes.c_void_p
    # gamma out of range: rejected before any CUDA call
    rc = lib.sdd_confidence(VP(16), 1, 1, 0, 100, 104, VP(16), VP(16), None, None, None, None, None, VP(256),
                            1 << 20, None, None)
    assert rc == 1 and b"gamma" in lib.sdd_last_error()
    # row stride not a multiple of 16 bytes
    rc = lib.sdd_confidence(VP(16), 1, 1, 4, 100, 100, VP(16), VP(16), None, None, None, None, None, VP(256),
                            1 << 20, None, None)
    assert rc == 1 and b"16 bytes" in lib.sdd_last_error()
    # n_tau out of range
    rc = lib.sdd_schedule_prefix(VP(16), None, 4, 8, 0, _f64_array([0.9]), _f64_array([0.9]), 0, 6, 64, None,
                                 None, None, VP(16), VP(16), None, None, None)
    assert rc == 1 and b"n_tau" in lib.sdd_last_error()
    # unknown signal
    rc = lib.sdd_schedule_prefix(VP(16), None, 4, 8, 7, _f64_array([0.9]), _f64_array([0.9]), 1, 6, 64, None,
                                 None, None, VP(16), VP(16), None, None, None)
    assert rc == 1 and b"signal" in lib.sdd_last_error()
    # lenience outside the paper's (0, 1] convention
    rc = lib.sdd_verify_lenient(VP(16), 1, 2, 4, 64, 64, VP(16), _f64_array([1.5]), 1, None, 2, VP(16), VP(16),
                                VP(16), VP(256), 1 << 20, None, None)
    assert rc == 1 and b"ell" in lib.sdd_last_error()
    # rows NULL with n_rows != B
    rc = lib.sdd_verify_topk(VP(16), 1, 2, 4, 64, 64, VP(16), (ctypes.c_int32 * 1)(2), 1, None, 1, VP(16),
                             VP(16), VP(16), VP(256), 1 << 20, None, None)
    assert rc == 1 and b"n_rows" in lib.sdd_last_error()


def test_status_from_device_rejects_null_on_host(lib):
    VP = ctypes.c_void_p
    bits = ctypes.c_uint32(7)
    assert lib.sdd_status_from_device(None, 0, ctypes.byref(bits), None) == 1
    assert b"NULL" in lib.sdd_last_error() and bits.value == 7
    assert lib.sdd_status_from_device(VP(16), 0, None, None) == 1


def test_scorer_workspace_size_and_check(lib):
    # 512 KiB per started 128-position tile: four split-K partials of 128 x 256 fp32
    n = ctypes.c_size_t(0)
    for M, tiles in ((0, 0), (1, 1), (128, 1), (129, 2), (4096, 32)):
        assert lib.sdd_scorer_workspace_size(M, ctypes.byref(n)) == 0
        assert n.value == tiles * 4 * 256 * 128 * 4
    assert lib.sdd_scorer_workspace_size(-1, ctypes.byref(n)) == 1
    assert lib.sdd_scorer_workspace_size(4, None) == 1
    # a workspace one byte short, or missing, is rejected before any CUDA call
    VP = ctypes.c_void_p
    need = 2 * 4 * 256 * 128 * 4
    rc = lib.sdd_survival_mlp(VP(16), 129, 64, VP(16), VP(16), VP(16), 0.0, VP(16), VP(256), need - 1, None, None)
    assert rc == 1 and b"workspace" in lib.sdd_last_error()
    rc = lib.sdd_survival_mlp(VP(16), 129, 64, VP(16), VP(16), VP(16), 0.0, VP(16), None, need, None, None)
    assert rc == 1 and b"workspace" in lib.sdd_last_error()
    rc = lib.sdd_scorer_deep(VP(16), 64, VP(16), 129, VP(16), VP(16), VP(16), VP(16), VP(16), VP(16), VP(16), 0.0,
                             VP(16), VP(16), VP(256), need - 1, None, None)
    assert rc == 1 and b"workspace" in lib.sdd_last_error()


def test_empty_batch_is_a_no_op(lib):
    VP = ctypes.c_void_p
    # B = 0 returns before touching the device or the workspace
    assert lib.sdd_confidence(None, 1, 0, 4, 100, 104, None, None, None, None, None, None, None, None, 0, None,
                              None) == 0
    assert lib.sdd_commit(None, None, None, None, 0, 4, None, None, None) == 0
    assert lib.sdd_agreement(None, None, 0, 3, None, None) == 0


def test_shard_record_layout_matches_c(tmp_path):
    """sdd_shard_partial is exchanged between ranks as plain bytes: 160 bytes,
    fields at fixed offsets."""
    from paper_2608_14787_gb300.vocab_shard import RECORD_BYTES
    want = {"m": 0, "r": 4, "t2": 8, "sh": 12, "sl": 16, "amax": 20, "g": 24, "info": 28, "cz": 32, "cv": 96}
    prog = ["#include <stdio.h>", "#include <stddef.h>", f'#include "{HEADER}"', "int main(void) {",
            'printf("%zu\\n", sizeof(sdd_shard_partial));']
    for f in want:
        prog.append(f'printf("%zu\\n", offsetof(sdd_shard_partial, {f}));')
    prog.append("return 0; }")
    c = tmp_path / "rec.c"
    c.write_text("\n".join(prog))
    exe = tmp_path / "rec"
    subprocess.check_call(["gcc", "-std=c11", "-o", str(exe), str(c)])
    vals = [int(x) for x in subprocess.check_output([str(exe)]).split()]
    assert vals[0] == RECORD_BYTES == 160
    assert dict(zip(want, vals[1:])) == want


def test_shard_arguments_rejected_on_host(lib):
    from paper_2608_14787_gb300.binding import BlockArgs
    a = BlockArgs()
    a.dtype, a.B, a.gamma, a.V, a.row_stride = 1, 2, 4, 1000, 504
    a.draft_logits = a.target_logits = a.draft_tokens = 256
    out = ctypes.c_void_p(256)
    # slice outside [0, V)
    assert lib.sdd_shard_partials(ctypes.byref(a), 900, 1001, out, None) == 1
    assert b"slice" in lib.sdd_last_error()
    # slice wider than the row stride
    assert lib.sdd_shard_partials(ctypes.byref(a), 0, 600, out, None) == 1
    # top-k beyond the candidates a record keeps
    ks = (ctypes.c_int32 * 1)(17)
    a.n_k, a.topk = 1, ctypes.cast(ks, ctypes.POINTER(ctypes.c_int32))
    assert lib.sdd_shard_partials(ctypes.byref(a), 0, 500, out, None) == 2
    # shard index out of range
    a.n_k = 0
    assert lib.sdd_shard_draw(ctypes.byref(a), 0, 500, 2, 2, ctypes.c_void_p(256), None) == 1
    n = ctypes.c_size_t(0)
    # per block: the 32-byte draw state, a counter, 64 segments' p_t masses and
    # 64 x 256 per-thread prefixes (each region 16-byte aligned)
    up = lambda v: (v + 15) // 16 * 16   # noqa: E731
    want = up(up(up(5 * 32) + 5 * 4) + 5 * 64 * 4) + 5 * 64 * 256 * 4
    assert lib.sdd_shard_workspace_size(5, ctypes.byref(n)) == 0 and n.value == want


def test_pipelined_arguments_rejected_on_host(lib):
    from paper_2608_14787_gb300.binding import BlockArgs
    assert lib.sdd_block_pipelined(None, None, None) == 1
    assert b"both NULL" in lib.sdd_last_error()
    a, b = BlockArgs(), BlockArgs()
    for x in (a, b):
        x.dtype, x.B, x.gamma, x.V, x.row_stride = 1, 2, 4, 1000, 1000
        x.draft_logits = x.target_logits = x.draft_tokens = 256
        x.workspace = 4096
    # two rounds in flight cannot share one workspace
    assert lib.sdd_block_pipelined(ctypes.byref(a), ctypes.byref(b), None) == 1
    assert b"workspace" in lib.sdd_last_error()
