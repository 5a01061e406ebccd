"""The C-ABI library loads, exports every declared entry point, and rejects bad
arguments on the host before touching the GPU (CPU only: no compute calls)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2606_09862_gb300 import build, bla
    build.build()
    return bla.load()


def declared_functions():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(bla_\w+)\s*\(", text))
    return sorted(names)


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert "bla_forward_chunked" in names and "bla_decode_step" in names and "bla_backward" in names
    for n in names:
        assert hasattr(lib, n), "missing export " + n


def test_status_strings(lib):
    assert lib.bla_status_string(0) == b"ok"
    assert lib.bla_status_string(4) == b"device wait timed out"


def _params(**kw):
    from paper_2606_09862_gb300 import bla
    base = dict(B=1, H=2, L=16, d_k=32, d_v=32, M=4, S=4, window=16.0, omega=0.0, chunk=0, scale=0.0,
                dtype=bla.BLA_F32)
    base.update(kw)
    return bla.Params(**base)


FAKE = ctypes.c_void_p(0x10000)      # aligned, never dereferenced: validation fails first


@pytest.mark.parametrize("kw", [dict(B=0), dict(H=0), dict(L=-1), dict(d_k=0), dict(M=0), dict(S=0),
                                dict(S=17), dict(window=0.0), dict(window=float("nan")), dict(dtype=7),
                                dict(chunk=-3), dict(omega=float("inf")), dict(phase_mode=2),
                                dict(phase_mode=-1)])
def test_invalid_params_rejected_on_host(lib, kw):
    from paper_2606_09862_gb300 import bla
    p = _params(**kw)
    st = lib.bla_forward_chunked(ctypes.byref(p), FAKE, FAKE, FAKE, FAKE, None, None, FAKE, 1 << 30, None)
    assert st == bla.BLA_ERR_INVALID
    assert lib.bla_last_error_string() != b""
    assert lib.bla_workspace_bytes(ctypes.byref(p), 0) == 0


def test_null_and_misaligned_pointers_rejected(lib):
    from paper_2606_09862_gb300 import bla
    p = _params()
    assert lib.bla_forward_chunked(None, FAKE, FAKE, FAKE, FAKE, None, None, FAKE, 1 << 30, None) == \
        bla.BLA_ERR_INVALID
    assert lib.bla_forward_chunked(ctypes.byref(p), None, FAKE, FAKE, FAKE, None, None, FAKE, 1 << 30, None) == \
        bla.BLA_ERR_INVALID
    bad = ctypes.c_void_p(0x10004)
    assert lib.bla_forward_chunked(ctypes.byref(p), bad, FAKE, FAKE, FAKE, None, None, FAKE, 1 << 30, None) == \
        bla.BLA_ERR_INVALID
    # workspace too small / misaligned
    assert lib.bla_forward_chunked(ctypes.byref(p), FAKE, FAKE, FAKE, FAKE, None, None, FAKE, 8, None) == \
        bla.BLA_ERR_INVALID
    assert lib.bla_forward_chunked(ctypes.byref(p), FAKE, FAKE, FAKE, FAKE, None, None,
                                   ctypes.c_void_p(0x10010), 1 << 30, None) == bla.BLA_ERR_INVALID


def test_decode_argument_checks(lib):
    from paper_2606_09862_gb300 import bla
    p = _params()
    assert lib.bla_decode_step(ctypes.byref(p), -1, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == \
        bla.BLA_ERR_INVALID
    p2 = _params(d_k=48, d_v=48)
    assert lib.bla_decode_step(ctypes.byref(p2), 0, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == \
        bla.BLA_ERR_UNSUPPORTED


def test_both_decode_entry_points_share_their_checks(lib):
    """bla_decode_step and bla_decode_step_noalloc reject the same arguments on the host, before any
    launch: B*H beyond the int grid, a negative position, an unsupported head size, and a mode count
    whose decode needs more shared memory than a CTA has."""
    from paper_2606_09862_gb300 import bla

    def both(p, pos=0):
        a = lib.bla_decode_step(ctypes.byref(p), pos, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 30, None)
        b = lib.bla_decode_step_noalloc(ctypes.byref(p), pos, FAKE, FAKE, FAKE, FAKE, FAKE, None)
        return a, b

    assert both(_params(B=1 << 16, H=1 << 16)) == (bla.BLA_ERR_INVALID,) * 2
    assert both(_params(), pos=-1) == (bla.BLA_ERR_INVALID,) * 2
    assert both(_params(d_k=48, d_v=48)) == (bla.BLA_ERR_UNSUPPORTED,) * 2
    assert both(_params(M=30000, S=64, window=1e5)) == (bla.BLA_ERR_UNSUPPORTED,) * 2
    assert b"shared memory" in lib.bla_last_error_string()


def test_workspace_sizes_positive(lib):
    from paper_2606_09862_gb300 import bla
    p = _params()
    assert lib.bla_workspace_bytes(ctypes.byref(p), bla.BLA_WS_FORWARD) > 0
    assert lib.bla_workspace_bytes(ctypes.byref(p), bla.BLA_WS_DECODE) > 0


def test_selftest_limit_checked_on_host(lib):
    from paper_2606_09862_gb300 import bla
    assert lib.bla_selftest_wait_timeout(0, None) == bla.BLA_ERR_INVALID
    assert lib.bla_selftest_wait_timeout(5000, None) == bla.BLA_ERR_INVALID


def test_host_forward_argument_checks(lib):
    """The host-buffer forward validates its arguments before any copy, and its workspace holds the
    forward's own plus the device copies of q, k, v and o."""
    from paper_2606_09862_gb300 import bla
    p = _params(dtype=bla.BLA_BF16, d_k=64, d_v=64, M=32, S=32, window=256.0, L=300)
    assert lib.bla_forward_chunked_host(ctypes.byref(p), None, FAKE, FAKE, FAKE, FAKE, 1 << 30, None) == \
        bla.BLA_ERR_INVALID
    assert lib.bla_forward_chunked_host(ctypes.byref(p), FAKE, FAKE, FAKE, FAKE, FAKE, 8, None) == bla.BLA_ERR_INVALID
    fw = lib.bla_workspace_bytes(ctypes.byref(p), bla.BLA_WS_FORWARD)
    hw = lib.bla_workspace_bytes(ctypes.byref(p), bla.BLA_WS_FORWARD_HOST)
    assert hw >= fw + 4 * 2 * 300 * 64 * 2


def test_phase_mode_accepted(lib):
    """Both phase modes are valid parameters; the absolute form's backward needs its per-chunk
    phase table on top of the lag form's workspace."""
    from paper_2606_09862_gb300 import bla
    for mode in (bla.BLA_PHASE_LAG, bla.BLA_PHASE_ABSOLUTE):
        p = _params(phase_mode=mode)
        assert lib.bla_workspace_bytes(ctypes.byref(p), bla.BLA_WS_FORWARD) > 0
        assert lib.bla_workspace_bytes(ctypes.byref(p), bla.BLA_WS_DECODE) > 0
    kw = dict(L=300, d_k=64, d_v=64, M=32, S=32, window=256.0, dtype=bla.BLA_BF16)
    lag = lib.bla_workspace_bytes(ctypes.byref(_params(**kw)), bla.BLA_WS_BACKWARD)
    ab = lib.bla_workspace_bytes(ctypes.byref(_params(phase_mode=bla.BLA_PHASE_ABSOLUTE, **kw)),
                                 bla.BLA_WS_BACKWARD)
    assert lag > 0 and ab > lag
    assert bla.make_params(1, 1, 8, 32, 32, 4, 4, 16.0, phase_mode="absolute").phase_mode == 1
    with pytest.raises(bla.BlaError):
        bla.make_params(1, 1, 8, 32, 32, 4, 4, 16.0, phase_mode="relative")


def test_product_path_does_not_import_oracle():
    """The CUDA binding and package never import the oracle."""
    pkg = os.path.join(ROOT, "paper_2606_09862_gb300")
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if fn.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, fn)).read()
                assert "import oracle" not in text and "from oracle" not in text, fn
                assert "bla_oracle" not in text and "liborc" not in text, fn


def test_decay_argument_checks(lib):
    """The state-decay entry points refuse the lag form, unsupported shapes and bad positions on the
    host, and size their workspace from the B*H*S*L slot scores."""
    from paper_2606_09862_gb300 import bla
    ab = bla.BLA_PHASE_ABSOLUTE

    def fwd(p, pos0=0, ws=1 << 30):
        return lib.bla_decay_forward(ctypes.byref(p), pos0, FAKE, FAKE, FAKE, FAKE, None, None, None, FAKE, ws, None)

    def dec(p, pos=0):
        return lib.bla_decay_decode_step(ctypes.byref(p), pos, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 30, None)

    assert fwd(_params()) == bla.BLA_ERR_UNSUPPORTED                     # lag form
    assert dec(_params()) == bla.BLA_ERR_UNSUPPORTED
    assert fwd(_params(phase_mode=ab), pos0=-1) == bla.BLA_ERR_INVALID
    assert dec(_params(phase_mode=ab), pos=-1) == bla.BLA_ERR_INVALID
    assert fwd(_params(phase_mode=ab, d_k=48, d_v=48)) == bla.BLA_ERR_UNSUPPORTED
    assert fwd(_params(phase_mode=ab, d_k=32, d_v=64)) == bla.BLA_ERR_UNSUPPORTED
    assert fwd(_params(phase_mode=ab, S=300, window=1000.0)) == bla.BLA_ERR_UNSUPPORTED
    assert fwd(_params(phase_mode=ab), ws=8) == bla.BLA_ERR_INVALID
    assert lib.bla_decay_forward(ctypes.byref(_params(phase_mode=ab)), 0, None, FAKE, FAKE, FAKE, None, None, None,
                                 FAKE, 1 << 30, None) == bla.BLA_ERR_INVALID
    p = _params(phase_mode=ab, B=2, H=3, L=100, S=8, window=40.0)
    assert lib.bla_workspace_bytes(ctypes.byref(p), bla.BLA_WS_DECAY_FORWARD) >= 2 * 3 * 8 * 100 * 4
    assert lib.bla_workspace_bytes(ctypes.byref(p), bla.BLA_WS_DECAY_DECODE) > 0
    assert lib.bla_workspace_bytes(ctypes.byref(_params()), bla.BLA_WS_DECAY_FORWARD) == 0
    bwd = lib.bla_decay_backward
    assert bwd(ctypes.byref(_params()), 0, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 30,
               None) == bla.BLA_ERR_UNSUPPORTED                                       # lag form
    assert bwd(ctypes.byref(_params(phase_mode=ab)), -1, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE,
               1 << 30, None) == bla.BLA_ERR_INVALID
    assert bwd(ctypes.byref(_params(phase_mode=ab)), 0, FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE,
               1 << 30, None) == bla.BLA_ERR_INVALID                                  # no lse
    assert lib.bla_workspace_bytes(ctypes.byref(p), bla.BLA_WS_DECAY_BACKWARD) >= 2 * 2 * 3 * 8 * 100 * 4
    # grids that would exceed the launch limits are refused before any launch
    assert fwd(_params(phase_mode=ab, B=1 << 20, H=1 << 10, S=64, window=64.0)) == bla.BLA_ERR_UNSUPPORTED


def test_per_head_periods_checked_on_host(lib):
    """Per-head periods (Alg. 1 and Alg. 3: T in R^H): each must be > 0, S must fit under all of
    them, at most 256 heads, and the paths without per-head tables refuse them before any launch."""
    from paper_2606_09862_gb300 import bla

    def params(periods, **kw):
        p = _params(H=len(periods), **kw)
        p.periods = (ctypes.c_double * len(periods))(*periods)
        return p

    def fwd(p):
        return lib.bla_forward_chunked(ctypes.byref(p), FAKE, FAKE, FAKE, FAKE, None, None, FAKE, 1 << 30, None)

    assert fwd(params([16.0, -1.0])) == bla.BLA_ERR_INVALID
    assert fwd(params([16.0, float("nan")])) == bla.BLA_ERR_INVALID
    assert fwd(params([16.0, 3.0], S=8, M=2)) == bla.BLA_ERR_INVALID          # S above one head's period
    assert fwd(params([16.0] * 257)) == bla.BLA_ERR_UNSUPPORTED
    p = params([16.0, 32.0])
    assert lib.bla_backward(ctypes.byref(p), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 30,
                            None) == bla.BLA_ERR_UNSUPPORTED
    # the tables repeat per head, so the workspace grows with H (decode, and the bf16 forward's
    # per-chunk EB tables)
    shared = lib.bla_workspace_bytes(ctypes.byref(_params(H=2)), bla.BLA_WS_DECODE)
    assert lib.bla_workspace_bytes(ctypes.byref(p), bla.BLA_WS_DECODE) > shared
    kw = dict(dtype=bla.BLA_BF16, d_k=64, d_v=64, M=32, S=32, L=4096)
    shared = lib.bla_workspace_bytes(ctypes.byref(_params(H=2, window=256.0, **kw)), bla.BLA_WS_FORWARD)
    per = lib.bla_workspace_bytes(ctypes.byref(params([256.0, 300.0], window=300.0, **kw)), bla.BLA_WS_FORWARD)
    assert per >= shared + 32 * 64 * 128 * 2      # a second copy of the 32 chunks' EB tables
    assert bla.make_params(1, 2, 8, 32, 32, 4, 4, [9.0, 20.0]).periods[1] == 20.0
    with pytest.raises(bla.BlaError):
        bla.make_params(1, 3, 8, 32, 32, 4, 4, [9.0, 20.0])
