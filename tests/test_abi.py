"""The C-ABI library builds, loads, exports every symbol include/qmla.h declares,
and validates arguments on the host (no GPU needed for any of this)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "qmla.h")


@pytest.fixture(scope="module")
def libqmla():
    import paper_2609_36760_gb300 as Q
    from paper_2609_36760_gb300 import build
    if not os.path.exists(Q.library_path()):
        build.build()
    return Q.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(qmla_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ["qmla_quant_append", "qmla_mla_decode", "qmla_mla_decode_bf16cache", "qmla_block_bytes",
                     "qmla_decode_workspace_bytes", "qmla_read_dev_err", "qmla_bf16_append"]:
        assert required in names


def test_library_exports_every_declared_symbol(libqmla):
    for name in declared_functions():
        assert hasattr(libqmla, name), name


def test_pure_host_queries(libqmla):
    assert libqmla.qmla_block_bytes(4) == 20736
    assert libqmla.qmla_block_bytes(2) == 12544
    assert libqmla.qmla_block_bytes(3) == 0 and libqmla.qmla_block_bytes(8) == 0
    assert libqmla.qmla_bf16_block_bytes() == 73728
    assert libqmla.qmla_status_string(0) == b"ok"
    assert libqmla.qmla_status_string(3) == b"workspace too small"


def test_invalid_arguments_are_rejected_before_any_launch(libqmla):
    L = libqmla
    fake = ctypes.c_void_p(0x10000)  # never dereferenced: validation fails first
    # bad bit width
    assert L.qmla_quant_append(fake, 3, 4, fake, fake, None, fake, 1, fake, 1, 1, None, None) == 1
    # null positions
    assert L.qmla_quant_append(fake, 4, 4, fake, fake, None, None, 1, fake, 1, 1, None, None) == 1
    # misaligned pool (32-byte alignment)
    assert L.qmla_quant_append(ctypes.c_void_p(0x10001), 4, 4, fake, fake, None, fake, 1, fake, 1, 1, None, None) == 1
    assert L.qmla_quant_append(ctypes.c_void_p(0x10010), 4, 4, fake, fake, None, fake, 1, fake, 1, 1, None, None) == 1
    # n == 0 is a no-op that touches nothing
    assert L.qmla_quant_append(None, 4, 4, None, None, None, None, 0, None, 1, 1, None, None) == 0
    # decode: heads out of range, null output, bad scale, bad bits
    args = [fake, 4, 4, fake, fake, 1, 129, fake, 1, fake, 0.1, fake, None, fake, 1 << 30, None, None]
    assert L.qmla_mla_decode(*args) == 1
    args[6] = 16
    args[11] = None
    assert L.qmla_mla_decode(*args) == 1
    args[11] = fake
    args[10] = -1.0
    assert L.qmla_mla_decode(*args) == 1
    args[10] = 0.1
    args[1] = 8
    assert L.qmla_mla_decode(*args) == 1
    assert L.qmla_decode_workspace_bytes(0, 16) == 0
    assert L.qmla_decode_workspace_bytes(1, 0) == 0


def test_c4r4_host_checks(libqmla):
    L = libqmla
    assert L.qmla_c4r4_page_bytes() == 20480
    fake = ctypes.c_void_p(0x10000)
    # protection rows asked for without the lengths after the call
    assert L.qmla_quant_append_c4r4(fake, 4, fake, fake, None, fake, 1, fake, 1, 1, None, fake, None, None) == 1
    # misaligned protection buffer
    assert L.qmla_quant_append_c4r4(fake, 4, fake, fake, None, fake, 1, fake, 1, 1, fake, ctypes.c_void_p(0x10008),
                                    None, None) == 1
    # n == 0: nothing to do, nothing touched
    assert L.qmla_quant_append_c4r4(None, 4, None, None, None, None, 0, None, 1, 1, None, None, None, None) == 0
    # decode: misaligned protection buffer, null output
    args = [fake, 4, fake, fake, 1, 16, fake, 1, fake, ctypes.c_void_p(0x10008), 0.1, fake, None, fake, 1 << 30,
            None, None]
    assert L.qmla_mla_decode_c4r4(*args) == 1
    args[9] = None
    args[11] = None
    assert L.qmla_mla_decode_c4r4(*args) == 1


def test_multi_query_host_checks(libqmla):
    L = libqmla
    assert L.qmla_decode_workspace_bytes(2, 128 * 8 + 1) == 0   # beyond 8 tokens x 128 heads
    fake = ctypes.c_void_p(0x10000)
    base = [fake, 4, 4, fake, fake, 1, 2, 16, fake, 1, fake, None, 0.1, fake, None, fake, 1 << 30, None, None]
    for i, bad in ((6, 0), (6, 9), (7, 0), (7, 129), (1, 3)):   # q_tokens, heads, c_bits
        args = list(base)
        args[i] = bad
        assert L.qmla_mla_decode_multi(*args) == 1, (i, bad)
    args = list(base)
    args[11] = ctypes.c_void_p(0x10008)                          # misaligned protection buffer
    assert L.qmla_mla_decode_multi(*args) == 1


def _desc(**kw):
    import paper_2609_36760_gb300 as Q
    fake = 0x10000
    d = Q.DecodeDesc()
    d.pool, d.cache_kind, d.num_blocks = fake, 4, 4
    d.q_latent, d.q_pe, d.batch, d.q_tokens, d.heads = fake, fake, 1, 1, 16
    d.block_table, d.max_blocks, d.seq_lens = fake, 1, fake
    d.prot, d.softmax_scale, d.out, d.lse = None, 0.1, fake, None
    d.workspace, d.workspace_bytes, d.dev_err = fake, 1 << 30, None
    for k, v in kw.items():
        setattr(d, k, v)
    return d


def test_decode_ex_host_checks(libqmla):
    L = libqmla
    assert L.qmla_mla_decode_ex(None, None) == 1                       # no descriptor
    for bad in ({"cache_kind": 3}, {"cache_kind": 8}, {"q_tokens": 0}, {"q_tokens": 9}, {"heads": 0},
                {"heads": 129}, {"batch": 0}, {"out": None}, {"workspace": None}, {"softmax_scale": -1.0},
                {"pool": 0x10008}, {"pool": 0x10010}, {"workspace": 0x10010}, {"prot": 0x10008},
                {"cache_kind": 16, "prot": 0x10000},                     # no protection on the BF16 cache
                {"cache_kind": 16, "q_tokens": 2}, {"cache_kind": 5, "q_tokens": 2}):
        d = _desc(**bad)
        assert L.qmla_mla_decode_ex(ctypes.byref(d), None) == 1, bad


def test_static_decode_host_checks(libqmla):
    # The allocation-free entry point rejects bad arguments before any device
    # call (so these run without a GPU): bits, heads, batch, pointers, scale,
    # alignment, table size.
    L = libqmla
    fake = ctypes.c_void_p(0x10000)
    base = [fake, 4, 4, fake, fake, 1, 16, fake, 1, fake, 0.1, fake, None, None, None]
    for i, bad in ((1, 3), (1, 8), (6, 0), (6, 129), (5, 0), (0, None), (3, None), (7, None), (9, None),
                   (11, None), (10, -1.0), (10, 0.0), (0, ctypes.c_void_p(0x10008)), (0, ctypes.c_void_p(0x10010)),
                   (3, ctypes.c_void_p(0x10004)), (11, ctypes.c_void_p(0x10004)), (8, 1 << 26)):
        args = list(base)
        args[i] = bad
        assert L.qmla_mla_decode_static(*args) == 1, (i, bad)


def test_debug_hooks_host_checks(libqmla):
    L = libqmla
    fake = ctypes.c_void_p(0x10000)
    assert L.qmla_debug_wait_timeout(0, fake, None) == 1          # limit below 1 us
    assert L.qmla_debug_wait_timeout(1000001, fake, None) == 1    # above 1 s
    assert L.qmla_debug_wait_timeout(10, None, None) == 1         # no error word
    # tile dump: bad kind, sequence outside the batch, tile beyond the table
    assert L.qmla_debug_tile(fake, 3, 4, fake, 2, fake, 1, 0, 0, None, fake, None, None) == 1
    assert L.qmla_debug_tile(fake, 4, 4, fake, 2, fake, 1, 1, 0, None, fake, None, None) == 1
    assert L.qmla_debug_tile(fake, 4, 4, fake, 2, fake, 1, 0, 1, None, fake, None, None) == 1


def test_trace_build_compiles(tmp_path):
    # The event-timeline variant of the decode (-DQMLA_TRACE_BUILD) is a separate
    # preprocessor path; compile it so it cannot rot unnoticed.
    import subprocess
    from paper_2609_36760_gb300 import build
    src = os.path.join(build.CSRC, "decode.cu")
    cmd = [build.nvcc(), *build.ARCH, *build.FLAGS, "-DQMLA_TRACE_BUILD", "-c", src, "-o", str(tmp_path / "d.o")]
    res = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    assert res.returncode == 0, res.stdout[-2000:]
