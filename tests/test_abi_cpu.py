"""The C ABI on a machine without a GPU: the library loads, exports every
entry point the header declares, and rejects bad arguments on the host
before any CUDA call is made."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "solo_readout.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(solo_readout_\w+)\s*\(", text)))


def test_header_declares_the_entry_points():
    names = declared_functions()
    for n in ("solo_readout_workspace_bytes", "solo_readout_fwd_bwd",
              "solo_readout_fwd_bwd_events", "solo_readout_get_flags",
              "solo_readout_strerror", "solo_readout_version"):
        assert n in names


def test_library_exports_every_declared_symbol(built_library):
    lib = ctypes.CDLL(built_library)
    for name in declared_functions():
        assert hasattr(lib, name), name


@pytest.fixture(scope="module")
def sr(built_library):
    from paper_2609_35440_gb300 import solo_readout
    solo_readout.load(built_library)
    return solo_readout


def test_strerror_and_version(sr):
    assert sr.strerror(0) == "success"
    for code in range(-6, 0):
        assert sr.strerror(code) and sr.strerror(code) != "unknown status"
    assert sr.strerror(-99) == "unknown status"
    assert sr.solo_readout_version() >= 100


def test_workspace_query(sr):
    dims = sr.make_dims(4, 8192, 2048, 32000)
    b = sr.solo_readout_workspace_bytes(dims)
    M = 4 * 8192
    # xhat (bf16) and the exponentials/gradient (bf16) dominate; the cut tiles
    # of the backward products take at most 32 MiB of fp32 partial tiles, and
    # no fp32 [K*N, d] buffer is reserved (it alone would be 268 MB here)
    assert b >= M * 2048 * 2 + M * 32000 * 2
    assert b < 1.05 * (M * 2048 * 2 + M * 32000 * 2) + 64 * 2 ** 20
    small = sr.solo_readout_workspace_bytes(sr.make_dims(1, 1, 8, 1))
    assert 0 < small < 2 ** 20


@pytest.mark.parametrize("K,N,d,V,want", [
    (0, 16, 64, 100, -1), (17, 16, 64, 100, -1), (2, 0, 64, 100, -1), (2, 16, 0, 100, -1),
    (2, 16, 64, 0, -1), (2, 16, 60, 100, -2), (2, 16, 4, 100, -1),
    # the largest vocabulary (the gradient pass keeps a float per 256-column tile
    # of a row in shared memory) and one past it
    (1, 16, 64, 1 << 23, 0), (1, 16, 64, (1 << 23) + 1, -2),
])
def test_workspace_query_rejects_bad_dims(sr, K, N, d, V, want):
    out = ctypes.c_size_t(0)
    st = sr.load().solo_readout_workspace_bytes(ctypes.byref(sr.make_dims(K, N, d, V)),
                                                ctypes.byref(out))
    assert st == want


def _args(sr, K=2, N=16, d=64, V=100, **over):
    fake = 1 << 20            # 16-byte aligned fake device addresses: never dereferenced
    a = dict(dims=sr.make_dims(K, N, d, V), hidden=[fake] * K, gamma=fake, W=fake,
             targets=fake, mask=None, loss_tok=None, loss_mean=fake, dhidden=[fake] * K,
             dW=None, dgamma=None, workspace=fake, workspace_bytes=1 << 40, stream=0)
    a.update(over)
    return a


@pytest.mark.parametrize("over,want", [
    (dict(gamma=None), -1), (dict(W=None), -1), (dict(targets=None), -1),
    (dict(loss_mean=None), -1), (dict(workspace=None), -1),
    (dict(hidden=[1 << 20, None]), -1), (dict(dhidden=[None, 1 << 20]), -1),
    (dict(W=(1 << 20) + 8), -6), (dict(hidden=[(1 << 20) + 2, 1 << 20]), -6),
    (dict(workspace=(1 << 20) + 4), -6), (dict(dW=(1 << 20) + 8), -6),
    (dict(workspace_bytes=1024), -3),
])
def test_fwd_bwd_rejects_bad_arguments_before_launch(sr, over, want):
    a = _args(sr, **over)
    st = sr.solo_readout_fwd_bwd(a["dims"], a["hidden"], a["gamma"], a["W"], a["targets"],
                                 a["mask"], a["loss_tok"], a["loss_mean"], a["dhidden"],
                                 a["dW"], a["dgamma"], a["workspace"],
                                 workspace_bytes=a["workspace_bytes"], stream=a["stream"],
                                 check=False)
    assert st == want


def test_fwd_bwd_rejects_bad_dims(sr):
    for dims, want in [(sr.make_dims(0, 16, 64, 100), -1), (sr.make_dims(2, 16, 12, 100), -2),
                       (sr.make_dims(2, 16, 64, 100, eps=-1.0), -1),
                       (sr.make_dims(2, 16, 64, 100, eps=float("nan")), -1)]:
        a = _args(sr, dims=dims)
        st = sr.solo_readout_fwd_bwd(dims, a["hidden"][:dims.K] or [1 << 20],
                                     a["gamma"], a["W"], a["targets"], None, None,
                                     a["loss_mean"], a["dhidden"][:dims.K] or [1 << 20], None,
                                     None, a["workspace"], workspace_bytes=1 << 40, stream=0,
                                     check=False) if dims.K > 0 else \
            sr.load().solo_readout_fwd_bwd(ctypes.byref(dims), None, None, None, None, None,
                                           None, None, None, None, None, None, 0, None)
        assert st == want


def test_events_variant_needs_all_events(sr):
    a = _args(sr)
    arr = (ctypes.c_void_p * 3)(1, 2, 3)
    st = sr._call(sr.load().solo_readout_fwd_bwd_events, a["dims"], a["hidden"], a["gamma"],
                  a["W"], a["targets"], None, None, a["loss_mean"], a["dhidden"], None, None,
                  a["workspace"], a["workspace_bytes"], 0, extra=(arr, 3))
    assert st == -1


def test_binding_has_no_fallback(tmp_path, monkeypatch):
    """A missing library raises instead of silently computing elsewhere."""
    from paper_2609_35440_gb300 import solo_readout
    monkeypatch.setattr(solo_readout, "_lib", None)
    with pytest.raises(ImportError):
        solo_readout.load(str(tmp_path / "missing.so"))


@pytest.mark.parametrize("flags,limit,want", [(None, 100, -1), (1 << 20, 0, -1),
                                              (1 << 20, 2000000, -1), ((1 << 20) + 2, 100, -6)])
def test_selftest_rejects_bad_arguments(sr, flags, limit, want):
    assert sr.solo_readout_selftest_wait_timeout(flags, limit, stream=0, check=False) == want


def test_exit_readout_host_checks(sr):
    fake = 1 << 20
    dims = sr.make_dims(2, 16, 64, 100)
    small = sr.solo_readout_exit_workspace_bytes(dims)
    assert 0 < small < sr.solo_readout_workspace_bytes(dims)
    # losses without targets, a missing hidden pointer, a small workspace
    assert sr.solo_readout_exit_forward(dims, [fake, fake], fake, fake, None, None, fake, None,
                                        fake, None, fake, workspace_bytes=1 << 30, stream=0,
                                        check=False) == sr.SOLO_ERR_INVALID_ARG
    assert sr.solo_readout_exit_forward(dims, [fake, None], fake, fake, fake, None, None, None,
                                        fake, None, fake, workspace_bytes=1 << 30, stream=0,
                                        check=False) == sr.SOLO_ERR_INVALID_ARG
    assert sr.solo_readout_exit_forward(dims, [fake, fake], fake, fake, fake, None, None, None,
                                        fake, None, fake, workspace_bytes=small - 1, stream=0,
                                        check=False) == sr.SOLO_ERR_WORKSPACE_TOO_SMALL


def test_private_host_checks(sr):
    fake = 1 << 20
    dims = sr.make_dims(3, 64, 64, 100)
    one = sr.solo_readout_private_workspace_bytes(dims)
    assert one < sr.solo_readout_workspace_bytes(dims)
    args = dict(hidden=[fake] * 3, gammas=[fake] * 3, Ws=[fake, fake, fake], targets=fake,
                mask=None, loss_tok=None, loss_mean=fake, dhidden=[fake] * 3, dWs=None,
                dgammas=None, workspace=fake, stream=0, check=False)
    assert sr.solo_readout_fwd_bwd_private(dims, **dict(args, Ws=[fake, None, fake]),
                                           workspace_bytes=one) == sr.SOLO_ERR_INVALID_ARG
    assert sr.solo_readout_fwd_bwd_private(dims, **args, workspace_bytes=one - 1) == \
        sr.SOLO_ERR_WORKSPACE_TOO_SMALL


def test_launch_counter_ignores_rejected_calls(sr):
    """Calls refused on the host enqueue nothing, so the counter stays put."""
    before = sr.solo_readout_kernel_launches()
    a = _args(sr, workspace_bytes=1024)
    assert sr.solo_readout_fwd_bwd(a["dims"], a["hidden"], a["gamma"], a["W"], a["targets"],
                                   None, None, a["loss_mean"], a["dhidden"], None, None,
                                   a["workspace"], workspace_bytes=1024, stream=0,
                                   check=False) == sr.SOLO_ERR_WORKSPACE_TOO_SMALL
    assert sr.solo_readout_kernel_launches() == before


def test_checked_build_exports_and_reports_itself(built_library):
    """The bounds-checked twin exports every declared symbol and says which it is."""
    from paper_2609_35440_gb300 import build as b
    path = b.LIB_CHECKED if b.up_to_date_checked() else b.build(checked=True)
    chk = ctypes.CDLL(path)
    for name in declared_functions():
        assert hasattr(chk, name), name
    assert chk.solo_readout_build_flags() == 1
    assert ctypes.CDLL(built_library).solo_readout_build_flags() == 0


def test_rmsnorm_host_checks(sr):
    fake = 1 << 20
    dims = sr.make_dims(2, 16, 64, 100)
    assert sr.solo_readout_rmsnorm(dims, [fake, None], fake, fake, stream=0,
                                   check=False) == sr.SOLO_ERR_INVALID_ARG
    assert sr.solo_readout_rmsnorm(dims, [fake, fake], fake, None, stream=0,
                                   check=False) == sr.SOLO_ERR_INVALID_ARG
    assert sr.solo_readout_rmsnorm(dims, [fake, fake], fake, fake + 8, stream=0,
                                   check=False) == sr.SOLO_ERR_MISALIGNED
    assert sr.solo_readout_rmsnorm(sr.make_dims(2, 16, 60, 100), [fake, fake], fake, fake,
                                   stream=0, check=False) == sr.SOLO_ERR_UNSUPPORTED_SHAPE


def test_overlapping_outputs_are_refused(sr):
    """An output that overlaps an input, another output or the workspace is
    refused before any launch; inputs may share memory."""
    base = 1 << 30
    K, N, d, V = 2, 16, 64, 100
    mb = 1 << 20
    ptr = {name: base + i * mb for i, name in enumerate(
        ["h0", "h1", "g", "W", "t", "lm", "dh0", "dh1", "dW", "dg", "lt", "ws"])}

    def call(**over):
        p = dict(ptr, **over)
        return sr.solo_readout_fwd_bwd(sr.make_dims(K, N, d, V), [p["h0"], p["h1"]], p["g"],
                                       p["W"], p["t"], None, p["lt"], p["lm"],
                                       [p["dh0"], p["dh1"]], p["dW"], p["dg"], p["ws"],
                                       workspace_bytes=1 << 40, stream=0, check=False)

    assert call(dW=ptr["W"]) == sr.SOLO_ERR_INVALID_ARG                 # output on an input
    assert call(dh0=ptr["h1"] + 256) == sr.SOLO_ERR_INVALID_ARG         # partial overlap
    assert call(dh1=ptr["dh0"]) == sr.SOLO_ERR_INVALID_ARG              # two outputs
    assert call(lm=ptr["ws"] + 4096) == sr.SOLO_ERR_INVALID_ARG         # inside the workspace
    # inputs sharing memory pass this check (the call then needs a GPU)
    assert call(h1=ptr["h0"]) != sr.SOLO_ERR_INVALID_ARG
    assert call() != sr.SOLO_ERR_INVALID_ARG


def test_exit_and_rmsnorm_overlaps_are_refused(sr):
    base, mb = 1 << 30, 1 << 20
    dims = sr.make_dims(2, 16, 64, 100)
    h0, h1, g, W, t, lt, lm, top, tlp, ws = (base + i * mb for i in range(10))
    exit_call = lambda **o: sr.solo_readout_exit_forward(
        dims, [h0, h1], g, W, t, None, o.get("lt", lt), lm, o.get("top", top), tlp, ws,
        workspace_bytes=1 << 40, stream=0, check=False)
    assert exit_call(top=W) == sr.SOLO_ERR_INVALID_ARG
    assert exit_call(lt=top) == sr.SOLO_ERR_INVALID_ARG
    assert exit_call() != sr.SOLO_ERR_INVALID_ARG
    assert sr.solo_readout_rmsnorm(dims, [h0, h1], g, h1, stream=0,
                                   check=False) == sr.SOLO_ERR_INVALID_ARG
    assert sr.solo_readout_rmsnorm(dims, [h0, h1], g, W, stream=0,
                                   check=False) != sr.SOLO_ERR_INVALID_ARG
