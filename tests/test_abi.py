"""The C-ABI library builds for sm_103a, loads, and exports every entry point that
include/fastmtp.h declares (no GPU needed: nothing is called).  Also the host-side argument
checks that return before any CUDA call."""
import ctypes
import os
import re

import pytest

from paper_2609_03181_gb300 import fastmtp as F

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "fastmtp.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return re.findall(r"^(?:spec_status|void|const char\*)\s+(\w+)\s*\(", src, flags=re.M)


def test_header_declares_the_binding_entry_points():
    assert declared_functions() == F.ENTRY_POINTS


def test_library_exports_every_declared_symbol():
    lib = F.load_library()
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_host_side_validation_without_gpu():
    lib = F.load_library()
    out = ctypes.c_void_p(123)
    # null config is rejected before any CUDA call, and *out is cleared
    assert lib.spec_init(None, None, None, None, None, ctypes.byref(out)) == F.SPEC_EINVAL
    assert out.value is None
    assert b"null" in lib.spec_last_error(None)
    cfg = F.SpecConfig(hidden=1024, n_heads=10, head_dim=128, n_layers=1, n_experts=64, top_k=6, n_shared=2,
                       expert_inter=896, draft_inter=3584, vocab=100, page_size=64, max_batch=1,
                       max_pages_per_seq=1, n_pages_total=1, K_max=3, max_position=64, rms_eps=1e-6,
                       rope_theta=1e6)
    w = F.SpecWeights()
    assert lib.spec_init(ctypes.byref(cfg), ctypes.byref(w), 16, 16, None, ctypes.byref(out)) == F.SPEC_EINVAL
    assert b"shape contract" in lib.spec_last_error(None)
    # every step rejects a NULL context
    assert lib.verify_step(None, 1, 0, None, None, None, None) == F.SPEC_EINVAL
    assert lib.draft_step(None, 1, 1, None, None) == F.SPEC_EINVAL
    assert lib.accept_commit(None, 1, None, None, None) == F.SPEC_EINVAL
    assert lib.spec_gemm_bf16(None, None, None, 1, 1, 64, None) == F.SPEC_EINVAL
    lib.spec_destroy(None)


def test_draft_loss_host_checks_without_gpu():
    lib = F.load_library()
    n = ctypes.c_size_t(5)
    assert lib.spec_draft_loss_workspace(0, 4, 100, ctypes.byref(n)) == F.SPEC_EINVAL and n.value == 0
    assert lib.spec_draft_loss_workspace(3, 64, 129280, None) == F.SPEC_EINVAL
    assert lib.spec_draft_loss_workspace(3, 64, 129280, ctypes.byref(n)) == F.SPEC_OK
    # packed rows 64 x 4 = 256 bf16 rows of 1280, 505 vocabulary tiles of 256 x 256 rows of 16-byte
    # partials, 3 x 64 x 3 floats; each part a multiple of 256 bytes
    assert n.value == 256 * 1280 * 2 + 505 * 256 * 16 + 2304
    assert lib.spec_draft_loss(None, None, None, None, None, 3, 4, 100, ctypes.c_float(0.6), ctypes.c_float(0.85),
                               ctypes.c_float(0.45), ctypes.c_float(0.45), None, None, None, 0, None) == F.SPEC_EINVAL
    assert b"null" in lib.spec_last_error(None)


def test_trace_read_without_the_timeline_build():
    # the normal build has no device timeline: spec_trace_read says so (no CUDA call), after its
    # argument checks
    lib = F.load_library()
    n = ctypes.c_int32(7)
    assert lib.spec_trace_read(None, 0, 1, None) == F.SPEC_EINVAL
    assert lib.spec_trace_read(None, 4, 1, ctypes.byref(n)) == F.SPEC_EINVAL   # NULL buffer with cap > 0
    assert lib.spec_trace_read(None, -1, 1, ctypes.byref(n)) == F.SPEC_EINVAL
    buf = (ctypes.c_uint64 * 8)()
    assert lib.spec_trace_read(buf, 2, 1, ctypes.byref(n)) == F.SPEC_EINVAL
    assert n.value == 0 and b"FASTMTP_TRACE" in lib.spec_last_error(None)
