"""The C ABI library without a GPU: it builds, loads, exports every symbol the
header declares, and its host-side validation rejects bad arguments before
anything is launched."""

import ctypes
import math
import os
import re

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2405_00263_gb300 import _lib, build
    build.build()
    return _lib.load()


def declared_symbols():
    names = []
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            names += re.findall(r"CLOVER_API\s+[\w\s\*]*?\b(clover_\w+)\s*\(", text)
    return names


def test_exports_every_declared_symbol(lib):
    from paper_2405_00263_gb300 import _lib
    names = declared_symbols()
    assert len(names) >= 7
    assert set(names) == set(_lib.EXPORTS)
    for n in names:
        assert hasattr(lib, n), n


def test_version_and_status_strings(lib):
    assert lib.clover_abi_version() == 1
    assert lib.clover_status_string(0) == b"ok"
    assert b"tree" in lib.clover_status_string(4)
    assert b"check" in lib.clover_status_string(128)
    assert lib.clover_build_flags() == 0          # the ordinary build compiles the device checks out


def test_workspace_sizes(lib):
    ws = lib.clover_verify_attn_workspace_size
    assert ws(1, 16, 8, 8, 64, 192, 0) == 0              # short cache: one split, no workspace
    big = ws(1, 64, 32, 32, 128, 4160, 0)                # fp32: CUDA-core split-KV merge
    assert big > 0 and big % 256 == 0
    # bf16 (tensor cores): 32 heads x 4 splits (one wave of 152 SMs) of 64 partial rows of
    # D + 4 floats, plus 32 arrival counters rounded up to 256 bytes
    assert ws(1, 64, 32, 32, 128, 4160, 1) == 32 * 4 * 64 * (128 + 4) * 4 + 256
    assert ws(4, 64, 64, 8, 128, 8256, 1) == 0            # 128 (head, row tile) groups: one split each
    assert ws(16, 32, 32, 32, 128, 8256, 1) == 0          # 512 heads: one split each
    assert ws(1, 129, 8, 8, 64, 192, 0) == 0             # T > 128 unsupported
    assert ws(1, 16, 8, 8, 96, 192, 0) == 0              # D = 96 unsupported
    assert ws(1, 16, 6, 4, 64, 192, 0) == 0              # Hq not a multiple of Hkv
    acc = lib.clover_verify_accept_workspace_size
    assert acc(1, 64, 125696, 1) == 8 * 64 + 4               # a 64-bit key per row, a counter per sequence
    assert acc(1, 0, 10, 1) == 0 and acc(1, 4, 0, 1) == 0


def _attn(lib, **kw):
    p = dict(q=16, k_new=16, v_new=16, kc=16, vc=16, cl=16, par=16, out=16, B=1, T=4, Hq=2, Hkv=2, D=64,
             Lcap=64, dt=1, scale=0.0, ws=None, wsb=0, st=None)
    p.update(kw)
    P = ctypes.c_void_p
    return lib.clover_verify_attn(P(p["q"]), P(p["k_new"]), P(p["v_new"]), P(p["kc"]), P(p["vc"]), P(p["cl"]),
                                  P(p["par"]), P(p["out"]), p["B"], p["T"], p["Hq"], p["Hkv"], p["D"], p["Lcap"],
                                  p["dt"], p["scale"], P(p["ws"]), p["wsb"], P(p["st"]), None)


def test_attn_host_validation(lib):
    # every case below returns before any CUDA call
    assert _attn(lib, T=129) == 2
    assert _attn(lib, D=80) == 2
    assert _attn(lib, Hq=3, Hkv=2) == 2
    assert _attn(lib, T=0) == 1
    assert _attn(lib, dt=7) == 1
    assert _attn(lib, Lcap=3) == 1
    assert _attn(lib, q=None) == 1
    assert _attn(lib, out=8) == 1                          # misaligned
    assert _attn(lib, scale=float("nan")) == 1
    assert _attn(lib, B=0) == 0                            # empty batch: nothing to do
    # fp32 needs a split-KV workspace at this size: refused before launch when it is missing
    assert _attn(lib, B=1, T=64, Hq=32, Hkv=32, D=128, Lcap=8192, dt=0, ws=None, wsb=0) == 1


def test_accept_and_compact_host_validation(lib):
    P = ctypes.c_void_p
    acc = lambda B, T, V, ws, wsb, lg=16: lib.clover_verify_accept(
        P(lg), P(16), P(16), B, T, V, 1, P(16), P(16), P(16), P(16), P(ws), wsb, None, None)
    assert acc(1, 129, 10, 16, 1 << 20) == 2
    assert acc(1, 4, 0, 16, 1 << 20) == 1
    assert acc(1, 4, 10, 16, 0) == 1                       # workspace too small
    assert acc(1, 4, 10, 16, 1 << 20, lg=17) == 1          # logits misaligned for bf16
    assert acc(0, 4, 10, None, 0) == 0
    cmp = lambda cl, ncl, B=2, T=4, D=64: lib.clover_kv_compact(
        P(16), P(16), P(cl), P(16), P(16), P(ncl), None, B, T, 2, D, 64, 1, None, None)
    assert cmp(1024, 1024) == 1                            # new length aliases the old one
    assert cmp(1024, 1028) == 1                            # partial overlap
    assert cmp(1024, 2048, D=32) == 2
    assert cmp(1024, 2048, T=129) == 2
    assert cmp(1024, 2048, B=0) == 0


def test_attn_ex_and_commit_host_validation(lib):
    P = ctypes.c_void_p
    ex = lambda flags, T=4: lib.clover_verify_attn_ex(
        P(16), P(16), P(16), P(16), P(16), P(16), P(16), P(16), 1, T, 2, 2, 64, 64, 1, 0.0, None, 0, None, None,
        flags)
    assert ex(16) == 1 and ex(0xFFFFFFF0) == 1            # unknown flag bits
    assert ex(15, T=129) == 2                                # the known bits (append off, PDL, cache/inputs ready)
    assert ex(1, T=129) == 2 and ex(0, T=129) == 2           # the limits of clover_verify_attn
    com = lambda cl, ncl, kn=16, vn=16, B=2, T=4, D=64: lib.clover_kv_commit(
        P(16), P(16), P(kn), P(vn), P(cl), P(16), P(16), P(ncl), None, B, T, 2, D, 64, 1, None, None)
    assert com(1024, 1024) == 1                            # new length aliases the old one
    assert com(1024, 2048, kn=None) == 1                   # k_new missing
    assert com(1024, 2048, vn=24) == 1                     # v_new misaligned
    assert com(1024, 2048, D=32) == 2
    assert com(1024, 2048, T=129) == 2
    assert com(1024, 2048, B=0) == 0


def test_accept_typical_workspace_and_host_validation(lib):
    P = ctypes.c_void_p
    # keys + counters (2*4*8 + 2*4 = 72 bytes, padded to 80), one 16-byte
    # (max, s, u) record per row and 16384-element chunk (8 for V = 125696
    # bf16), one fp32 candidate logit per node
    need = lib.clover_verify_accept_typical_workspace_size(2, 4, 125696, 1)
    assert lib.clover_verify_accept_workspace_size(2, 4, 125696, 1) == 72
    assert need == 80 + 16 * 2 * 4 * 8 + 4 * 2 * 4
    assert lib.clover_verify_accept_typical_workspace_size(2, 4, 125696, 0) == 80 + 16 * 2 * 4 * 16 + 4 * 2 * 4
    assert lib.clover_verify_accept_typical_workspace_size(2, 129, 100, 1) == 0
    call = lambda tau=1.0, eps=0.09, delta=0.3, ws=4096, wsb=need, B=2, T=4, V=125696: \
        lib.clover_verify_accept_typical(P(64), P(64), P(64), B, T, V, 1, tau, eps, delta, P(64), P(64), P(64),
                                         P(64), P(ws), wsb, None, None)
    for bad in (dict(tau=0.0), dict(tau=-1.0), dict(tau=math.nan), dict(tau=math.inf), dict(eps=-0.1),
                dict(eps=math.nan), dict(delta=-1.0), dict(delta=math.inf), dict(ws=4104), dict(wsb=need - 1),
                dict(ws=0)):
        assert call(**bad) == 1, bad
    assert call(tau=1e-300) == 2 and call(tau=1e39) == 2     # log2(e)/tau not a normal fp32 number
    assert call(T=129) == 2
    assert call(B=0) == 0


def test_accept_ex_host_validation(lib):
    P = ctypes.c_void_p
    assert lib.clover_verify_accept_ex_workspace_size(2, 4, 125696, 1, 0) == \
        lib.clover_verify_accept_workspace_size(2, 4, 125696, 1)
    assert lib.clover_verify_accept_ex_workspace_size(2, 4, 125696, 1, 1) == \
        lib.clover_verify_accept_typical_workspace_size(2, 4, 125696, 1)

    def call(flags, tau=1.0, kn=64, D=128, B=2, T=4, ncl=4096, cl=2048, ws=4096):
        return lib.clover_verify_accept_ex(P(64), P(64), P(64), B, T, 1000, 1, tau, 0.09, 0.3, P(64), P(64), P(kn),
                                           P(64), P(cl), 2, D, 64, P(64), P(64), P(64), P(64), P(ncl), None, P(ws),
                                           1 << 20, flags, None, None)
    assert call(8) == 1 and call(0xFFFFFFF0) == 1             # unknown flag bits
    assert call(1, tau=0.0) == 1                             # typical: temperature must be > 0
    assert call(2, kn=0) == 1                                # commit: k_new missing
    assert call(2, kn=72) == 1                               # commit: k_new misaligned
    assert call(2, D=96) == 2                                # commit: D not 64/128
    assert call(2, ncl=2048) == 1                            # commit: new length aliases the old one
    assert call(1, ws=4104) == 1                             # typical: workspace 16-byte aligned
    assert call(7, T=129) == 2
    assert call(7, B=0) == 0


def test_paged_host_validation(lib):
    P = ctypes.c_void_p
    pw = lib.clover_verify_attn_paged_workspace_size
    assert pw(1, 64, 32, 32, 128, 64, 65, 0) == lib.clover_verify_attn_workspace_size(1, 64, 32, 32, 128, 64 * 65, 0)
    assert pw(1, 16, 8, 8, 64, 24, 10, 0) == 0 and pw(1, 16, 8, 8, 64, 8, 10, 0) == 0   # page 24, page 8
    assert pw(1, 16, 8, 8, 64, 2048, 10, 0) == 0 and pw(1, 16, 8, 8, 64, 64, 0, 0) == 0

    def attn(ps=64, n_pages=10, bt=64, T=4, B=1, D=64):
        return lib.clover_verify_attn_paged(P(64), P(64), P(64), P(64), P(64), P(bt), n_pages, ps, 8, P(64), P(64),
                                            P(64), B, T, 2, 2, D, 1, 0.0, None, 0, None, None)
    assert attn(ps=24) == 1 and attn(ps=8) == 1 and attn(n_pages=0) == 1 and attn(bt=0) == 1
    assert attn(T=129) == 2 and attn(D=96) == 2
    assert attn(B=0) == 0

    def commit(ps=64, bt=64, D=64, B=2, kn=64):
        return lib.clover_kv_commit_paged(P(64), P(64), P(bt), 10, ps, 8, P(kn), P(64), P(1024), P(64), P(64),
                                          P(2048), None, B, 4, 2, D, 1, None, None)
    assert commit(ps=100) == 1 and commit(bt=0) == 1 and commit(kn=0) == 1
    assert commit(D=96) == 2
    assert commit(B=0) == 0


def test_paged_ex_host_validation(lib):
    P = ctypes.c_void_p

    def attn(flags, ps=64, bt=64, T=4, B=1):
        return lib.clover_verify_attn_paged_ex(P(64), P(64), P(64), P(64), P(64), P(bt), 10, ps, 8, P(64), P(64),
                                               P(64), B, T, 2, 2, 64, 1, 0.0, None, 0, None, None, flags)
    assert attn(16) == 1 and attn(0xFFFFFFF0) == 1            # unknown flag bits
    assert attn(2, ps=24) == 1 and attn(8 | 2, bt=0) == 1
    assert attn(2, T=129) == 2
    assert attn(1 | 2 | 4 | 8, B=0) == 0                     # every known bit, NO_APPEND included

    def accept(flags, ps=64, bt=64, kn=64, D=64, B=2, T=4, ncl=4096, tau=1.0):
        return lib.clover_verify_accept_paged_ex(P(64), P(64), P(64), B, T, 1000, 1, tau, 0.09, 0.3, P(64), P(64),
                                                 P(bt), 10, ps, 8, P(kn), P(64), P(2048), 2, D, P(64), P(64), P(64),
                                                 P(64), P(ncl), None, P(4096), 1 << 20, flags, None, None)
    assert accept(8) == 1 and accept(0xFFFFFFF0) == 1        # unknown flag bits
    assert accept(2, ps=100) == 1 and accept(2, ps=8) == 1   # page size: a power of two >= 16
    assert accept(2, bt=0) == 1 and accept(0, kn=0) == 1     # block table, k_new (commit implied)
    assert accept(2, ncl=2048) == 1                          # new length aliases the old one
    assert accept(1, tau=0.0) == 1
    assert accept(2, D=96) == 2 and accept(2, T=129) == 2
    assert accept(7, B=0) == 0


def test_draft_host_validation(lib):
    P = ctypes.c_void_p
    lin = lambda R=4, N=128, K=64, mode=1, x=64, res=None, out=128, ws=None: lib.clover_linear(
        P(x), P(64), P(res) if res else None, P(out), R, N, K, mode, P(ws) if ws else None, 1 << 20, None, None)
    assert lin(ws=72) == 1                                   # workspace 16-byte aligned
    # 4096 x 4096: 32 tiles, 16 pairs -> 8 K ranges; partials of 16 rows and 4 counters a pair
    assert lib.clover_linear_workspace_size(16, 4096, 4096) == 8 * 16 * 4096 * 4 + 4 * 4 * 16
    assert lib.clover_linear_workspace_size(16, 125696, 4096) == 0     # enough tiles: no split
    assert lib.clover_linear_workspace_size(300, 256, 128) == 0         # under 4 stages of K per range: no split
    assert lin(K=96) == 1 and lin(K=0) == 1 and lin(N=0) == 1 and lin(mode=4) == 1 and lin(mode=-1) == 1
    assert lin(mode=2) == 1 and lin(mode=3) == 1             # residual modes need res
    assert lin(x=72) == 1 and lin(out=136) == 1              # 16-byte alignment
    assert lin(R=0) == 0
    lin_ex = lambda flags, R=4, K=64: lib.clover_linear_ex(P(64), P(64), None, P(128), R, 128, K, 1, flags, None, 0,
                                                           None, None)
    assert lin_ex(2) == 1 and lin_ex(0xFFFFFFFE) == 1        # unknown flag bits
    assert lin_ex(1, K=96) == 1 and lin_ex(1, R=0) == 0      # the same checks as clover_linear
    assert lib.clover_topk_workspace_size(3, 1000, 8) == 8 * 3 * 1 * 8 + 4 * 3
    assert lib.clover_topk_workspace_size(3, 125696, 8) == 8 * 3 * 16 * 8 + 4 * 3
    assert lib.clover_topk_workspace_size(1, 100, 33) == 0 and lib.clover_topk_workspace_size(1, 4, 5) == 0
    tk = lambda R=2, V=1000, k=4, ws=64, wsb=1 << 20: lib.clover_topk(P(64), R, V, k, P(64), P(64), P(ws), wsb,
                                                                     None, None)
    assert tk(k=0) == 1 and tk(k=1001) == 1 and tk(k=33) == 2
    assert tk(V=200000, k=32) == 2                          # 25 chunks x 32 candidates > 512
    assert tk(ws=68) == 1 and tk(wsb=8) == 1
    assert tk(R=0) == 0
    emb = lambda R=2, V=10, H=8: lib.clover_embed_rows(P(64), P(64), P(64), R, V, H, None, None)
    assert emb(V=0) == 1 and emb(H=0) == 1 and emb(R=-1) == 1 and emb(R=0) == 0


def test_python_binding_rejects_cpu_tensors(lib):
    import paper_2405_00263_gb300 as pkg
    x = torch.zeros(1, 4, 2, 64, dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        pkg.clover_verify_attn(x, x, x, torch.zeros(1, 2, 64, 64, dtype=torch.bfloat16),
                               torch.zeros(1, 2, 64, 64, dtype=torch.bfloat16), torch.zeros(1, dtype=torch.int32),
                               torch.zeros(1, 4, dtype=torch.int32), x.clone())


def test_oracle_and_library_share_no_code():
    """The oracle is plain C with its own definitions; the library sources never
    include or import anything under oracle/, and the oracle never reads csrc/."""
    csrc = os.path.join(ROOT, "paper_2405_00263_gb300", "csrc")
    for fn in os.listdir(csrc):
        assert "oracle" not in open(os.path.join(csrc, fn)).read().lower(), fn
    for fn in ("api.py", "_lib.py", "build.py", "__init__.py"):
        assert "import oracle" not in open(os.path.join(ROOT, "paper_2405_00263_gb300", fn)).read()
    src = open(os.path.join(ROOT, "oracle", "clover_oracle.c")).read()
    assert "#include \"" not in src and "clover_verify.h" not in src


def test_checked_build_exports_the_same_symbols():
    """The -DCLOVER_CHECKED variant builds, exports the declared symbols and
    reports itself through clover_build_flags (host-only calls)."""
    import ctypes
    from paper_2405_00263_gb300 import _lib
    from paper_2405_00263_gb300 import build as _build
    path = _build.build(checked=True)
    assert path == _build.CHECKED_LIB != _build.LIB
    lib = ctypes.CDLL(path)
    for n in declared_symbols():
        assert hasattr(lib, n), n
    assert lib.clover_build_flags() & _lib.BUILD_CHECKED


def test_verify_step_outputs_are_views_of_one_buffer(monkeypatch):
    """VerifyStep's host-side set-up without a GPU (streams, events and the
    workspace-size calls stubbed): every output is a contiguous, 16-byte
    aligned view of one buffer, and `results` spans exactly out, path,
    accept_len, bonus and new_cache_len."""
    from paper_2405_00263_gb300 import api

    class FakeStream:
        def __init__(self, *args, **kwargs):
            pass

        @staticmethod
        def priority_range():
            return (0, -1)

    monkeypatch.setattr(api, "clover_verify_attn_workspace_size", lambda *a: 0)
    monkeypatch.setattr(api, "clover_verify_accept_workspace_size", lambda *a: 64)
    monkeypatch.setattr(torch.cuda, "Stream", FakeStream)
    monkeypatch.setattr(torch.cuda, "Event", lambda *a, **k: None)
    B, T, Hq, D = 3, 37, 8, 128
    st = api.VerifyStep(B, T, Hq, 8, D, 512, 1000, torch.bfloat16, device="cpu")
    base = st._outputs.data_ptr()
    names = ["out", "path", "accept_len", "bonus", "new_cache_len", "argmax", "src_index"]
    shapes = [(B, T, Hq, D), (B, T), (B,), (B,), (B,), (B, T), (B, T)]
    spans = []
    for name, shape in zip(names, shapes):
        t = getattr(st, name)
        assert tuple(t.shape) == shape and t.is_contiguous() and t.data_ptr() % 16 == 0, name
        lo = t.data_ptr() - base
        spans.append((lo, lo + t.numel() * t.element_size()))
    assert all(a[1] <= b[0] for a, b in zip(spans, spans[1:]))      # disjoint, in order
    assert st.results.data_ptr() == base and st.results.numel() == spans[4][1]
