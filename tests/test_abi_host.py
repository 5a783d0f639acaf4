"""The C ABI without a GPU: the library loads, exports every declared entry point,
and rejects bad arguments before touching CUDA."""
import ctypes as C
import re
import shutil
import subprocess
from pathlib import Path

import pytest

import paper_2605_16941_gb300 as wino
from paper_2605_16941_gb300 import _abi

HEADER = Path(__file__).resolve().parents[1] / "include" / "wino.h"


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2605_16941_gb300 import build
    build.build()


def declared_functions():
    text = HEADER.read_text()
    return re.findall(r"WINO_API\s+[\w\s\*]+?\b(wino_\w+)\s*\(", text)


def test_every_declared_symbol_is_exported():
    names = declared_functions()
    assert set(names) == set(_abi.EXPORTS), names
    L = C.CDLL(str(wino.library_path()))
    for n in names:
        assert hasattr(L, n), n


def test_status_strings_and_version():
    assert wino.wino_version() == 1
    for code in (0, -1, -2, -3, -4, -5, -6, -7):
        assert wino.wino_status_string(code) != "unknown status"
    assert wino.wino_status_string(12345) == "unknown status"


def test_workspace_size():
    n = wino.wino_workspace_size(256, 4096, 126464)
    assert n >= 256 * 256 * 16 and n % 256 == 0  # at most 256 partial records per row
    for bad in ((0, 64, 100), (64, 60, 100), (64, 4, 100), (64, 64, 1), (1 << 25, 64, 100), (64, 64, 1 << 28)):
        with pytest.raises(wino.WinoError) as e:
            wino.wino_workspace_size(*bad)
        assert e.value.status == wino.WINO_ERR_SHAPE


FAKE = 0x10000  # 16-byte (and 256-byte) aligned, never dereferenced: every call below fails its checks first


def _p(**kw):
    base = dict(tau1=0.7, tau2=0.9, mask_id=99, n_seq=2, seq_len=64, blk_start=32, blk_len=16, max_steps=10,
                options=0)
    base.update(kw)
    return _abi.WinoParams(**base)


def test_score_rows_argument_errors():
    L = wino.lib()
    ok = dict(H=FAKE, W=FAKE, N=64, d=64, V=100, t=None, a=FAKE, pm=FAKE, pt=FAKE, ent=None, ws=FAKE, wsb=1 << 20,
              s=None)

    def call(**kw):
        a = dict(ok, **kw)
        return L.wino_score_rows(a["H"], a["W"], a["N"], a["d"], a["V"], a["t"], a["a"], a["pm"], a["pt"], a["ent"],
                                 a["ws"], a["wsb"], a["s"])
    for k in ("H", "W", "a", "pm", "pt", "ws"):
        assert call(**{k: None}) == wino.WINO_ERR_ARG, k
    assert call(H=FAKE + 2) == wino.WINO_ERR_ARG
    for k in ("a", "pm", "pt"):
        assert call(**{k: FAKE + 2}) == wino.WINO_ERR_ARG, k
    assert call(t=FAKE + 1) == wino.WINO_ERR_ARG
    assert call(ent=FAKE + 6) == wino.WINO_ERR_ARG
    assert call(W=FAKE + 8) == wino.WINO_ERR_ARG
    assert call(ws=FAKE + 16) == wino.WINO_ERR_ARG
    assert call(d=60) == wino.WINO_ERR_SHAPE
    assert call(N=0) == wino.WINO_ERR_SHAPE
    assert call(V=1) == wino.WINO_ERR_SHAPE


def test_draft_verify_argument_errors():
    L = wino.lib()

    def call(p, **kw):
        a = dict(tok=FAKE, am=FAKE, pm=FAKE, pt=FAKE, cnt=FAKE)
        a.update(kw)
        return L.wino_draft_verify(a["tok"], a["am"], a["pm"], a["pt"], C.byref(p) if p is not None else None,
                                   a["cnt"], None, None)
    for k in ("tok", "am", "pm", "pt", "cnt"):
        assert call(_p(), **{k: None}) == wino.WINO_ERR_ARG, k
    assert call(None) == wino.WINO_ERR_ARG
    assert call(_p(tau1=1.5)) == wino.WINO_ERR_ARG
    assert call(_p(tau2=-0.1)) == wino.WINO_ERR_ARG
    assert call(_p(tau1=float("nan"))) == wino.WINO_ERR_ARG
    assert call(_p(blk_len=0)) == wino.WINO_ERR_SHAPE
    assert call(_p(blk_len=1025, seq_len=2000)) == wino.WINO_ERR_SHAPE
    assert call(_p(blk_start=50)) == wino.WINO_ERR_SHAPE  # block runs past seq_len
    assert call(_p(n_seq=0)) == wino.WINO_ERR_SHAPE
    assert call(_p(mask_id=-1)) == wino.WINO_ERR_SHAPE
    assert call(_p(draft_m=-1)) == wino.WINO_ERR_ARG
    assert call(_p(active_seq=FAKE, n_active=1)) == wino.WINO_ERR_ARG  # the caller's rows: no list
    for k in ("tok", "am", "pm", "pt", "cnt"):
        assert call(_p(), **{k: FAKE + 2}) == wino.WINO_ERR_ARG, k
    assert call(_p(last_change=FAKE + 3)) == wino.WINO_ERR_ARG


def test_step_argument_errors():
    L = wino.lib()

    def call(p, d=64, V=100, wsb=1 << 30, **kw):
        a = dict(H=FAKE, W=FAKE, tok=FAKE, cnt=FAKE, ws=FAKE)
        a.update(kw)
        return L.wino_step(a["H"], a["W"], d, V, a["tok"], C.byref(p), a["cnt"], None, a["ws"], wsb, None)
    for k in ("H", "W", "tok", "cnt", "ws"):
        assert call(_p(), **{k: None}) == wino.WINO_ERR_ARG, k
    assert call(_p(mask_id=100)) == wino.WINO_ERR_SHAPE  # MASK outside the vocabulary
    assert call(_p(), d=12) == wino.WINO_ERR_SHAPE
    assert call(_p(), wsb=1000) == wino.WINO_ERR_WORKSPACE
    assert call(_p(), tok=FAKE + 2) == wino.WINO_ERR_ARG
    assert call(_p(), cnt=FAKE + 1) == wino.WINO_ERR_ARG
    assert call(_p(last_change=FAKE + 2)) == wino.WINO_ERR_ARG
    assert call(_p(active_seq=FAKE + 2, n_active=1)) == wino.WINO_ERR_ARG  # misaligned list
    assert call(_p(active_seq=FAKE, n_active=0)) == wino.WINO_ERR_SHAPE
    assert call(_p(active_seq=FAKE, n_active=3)) == wino.WINO_ERR_SHAPE  # more entries than sequences (2)


def test_params_layout_matches_header(tmp_path):
    """The ctypes mirror of wino_params has the C struct's size and field offsets (gcc reads the header)."""
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    fields = [f[0] for f in _abi.WinoParams._fields_]
    src = tmp_path / "layout.c"
    src.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "wino.h"\nint main(void) {\n'
                   '    printf("%zu\\n", sizeof(wino_params));\n' +
                   "".join('    printf("%%zu\\n", offsetof(wino_params, %s));\n' % f for f in fields) +
                   "    return 0;\n}\n")
    exe = tmp_path / "layout"
    inc = Path(__file__).resolve().parent.parent / "include"
    subprocess.run([gcc, "-std=c11", "-I", str(inc), str(src), "-o", str(exe)], check=True)
    got = [int(x) for x in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    assert got[0] == C.sizeof(_abi.WinoParams)
    assert got[1:] == [getattr(_abi.WinoParams, f).offset for f in fields]


def test_decode_argument_errors():
    """wino_decode refuses bad arguments before calling the hidden-state callback or launching anything."""
    L = wino.lib()
    called = []
    fn = _abi.HIDDEN_FN(lambda user, k, b0: called.append(k) or FAKE)
    host = (C.c_int32 * 6)()

    def call(p, n_blocks=2, first_block=0, first_step=0, hidden=fn, **kw):
        a = dict(W=FAKE, tok=FAKE, cnt=FAKE, cnth=C.addressof(host), fl=None, flh=None, act=None, ws=FAKE)
        a.update(kw)
        return L.wino_decode(a["W"], 64, 100, a["tok"], C.byref(p) if p is not None else None, n_blocks,
                             first_block, first_step, hidden, None, a["cnt"], a["cnth"], a["fl"], a["flh"], a["act"],
                             a["ws"], 1 << 30, None, None, None)
    for k in ("W", "tok", "cnt", "cnth", "ws"):
        assert call(_p(), **{k: None}) == wino.WINO_ERR_ARG, k
    assert call(None) == wino.WINO_ERR_ARG
    assert call(_p(), hidden=_abi.HIDDEN_FN()) == wino.WINO_ERR_ARG  # null callback
    assert call(_p(), n_blocks=0) == wino.WINO_ERR_ARG
    assert call(_p(), first_block=3) == wino.WINO_ERR_ARG
    assert call(_p(), first_step=-1) == wino.WINO_ERR_ARG
    assert call(_p(max_steps=0)) == wino.WINO_ERR_ARG
    assert call(_p(), n_blocks=3) == wino.WINO_ERR_SHAPE  # blocks 32..80 run past seq_len 64
    assert call(_p(), flh=C.addressof(host)) == wino.WINO_ERR_ARG  # host flags without device flags
    assert call(_p(active_seq=FAKE, n_active=1)) == wino.WINO_ERR_ARG  # the loop keeps its own list
    assert called == []
