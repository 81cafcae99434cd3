"""The C ABI without a GPU: every declared entry point is exported, and host-side
argument checks reject bad calls before any CUDA work (so they run on a CPU machine)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "chronostitch.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(cs_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_four_steps():
    names = declared_functions()
    for n in ("cs_rebase_keys", "cs_score_deviation", "cs_select_topk", "cs_repair_attention",
              "cs_sync_status", "cs_status_string"):
        assert n in names


def test_library_exports_every_declared_symbol(cslib):
    out = subprocess.run(["nm", "-D", "--defined-only", cslib.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\s[TW]\s+(\S+)", out))
    missing = [n for n in declared_functions() if n not in exported]
    assert not missing, missing
    handle = ctypes.CDLL(cslib.LIB_PATH)
    for n in declared_functions():
        assert getattr(handle, n) is not None


def test_status_strings(cslib):
    L = cslib.lib()
    assert cslib.cs_abi_version() == 1
    for code in range(6):
        assert L.cs_status_string(code)
    assert cslib.cs_status_string(0) == "ok"
    assert "timed out" in cslib.cs_status_string(4)


def _rope(theta=1e6, sec=(16, 24, 24)):
    import paper_2607_19547_gb300 as cs
    return cs._RopeCfg(theta, (ctypes.c_int32 * 3)(*sec))


FAKE = 1 << 20   # aligned non-null address: never dereferenced when validation fails


def test_rebase_rejects_bad_arguments(cslib):
    L = cslib.lib()
    r = _rope()

    def call(**kw):
        a = dict(k_in=FAKE, k_out=FAKE, dt=1, L=2, stride=4 * 2 * 128, T=4, H=2, D=128,
                 pl=FAKE, pg=FAKE, rope=ctypes.byref(r))
        a.update(kw)
        return L.cs_rebase_keys(a["k_in"], a["k_out"], a["dt"], a["L"], a["stride"], a["T"],
                                a["H"], a["D"], a["pl"], a["pg"], a["rope"], None)

    assert call(D=64) == cslib.CS_ERR_UNSUPPORTED
    assert "head_dim" in cslib.cs_last_error_detail()
    assert call(dt=7) == cslib.CS_ERR_INVALID_ARG
    assert call(T=-1) == cslib.CS_ERR_INVALID_ARG
    assert call(stride=100) == cslib.CS_ERR_INVALID_ARG
    bad = _rope(sec=(16, 24, 23))
    assert call(rope=ctypes.byref(bad)) == cslib.CS_ERR_INVALID_ARG
    assert "sections" in cslib.cs_last_error_detail()
    neg = _rope(sec=(-8, 48, 24))
    assert call(rope=ctypes.byref(neg)) == cslib.CS_ERR_INVALID_ARG
    low = _rope(theta=1.0)
    assert call(rope=ctypes.byref(low)) == cslib.CS_ERR_INVALID_ARG
    assert call(rope=None) == cslib.CS_ERR_INVALID_ARG
    assert call(k_in=None) == cslib.CS_ERR_INVALID_ARG
    assert call(k_in=FAKE + 8, k_out=FAKE + 8) == cslib.CS_ERR_INVALID_ARG     # misaligned
    assert call(k_out=FAKE + 256) == cslib.CS_ERR_INVALID_ARG                  # partial overlap
    assert call(H=40) == cslib.CS_ERR_UNSUPPORTED
    # coordinates are read while other CTAs write the keys
    far = FAKE + (1 << 24)
    assert call(pl=far, pg=FAKE + 512) == cslib.CS_ERR_INVALID_ARG
    assert "coordinates overlap" in cslib.cs_last_error_detail()
    assert call(pl=FAKE + 512, pg=far) == cslib.CS_ERR_INVALID_ARG
    assert "coordinates overlap" in cslib.cs_last_error_detail()
    # nothing to do: succeeds without touching the device
    assert call(L=0, k_in=None, k_out=None) == cslib.CS_OK
    assert call(T=0, k_in=None, k_out=None, stride=0) == cslib.CS_OK


def test_score_rejects_bad_arguments(cslib):
    L = cslib.lib()

    def call(**kw):
        a = dict(f=FAKE, c=FAKE, dt=1, n=5, H=2, D=128, fs=256, cs=256, out=FAKE)
        a.update(kw)
        return L.cs_score_deviation(a["f"], a["c"], a["dt"], a["n"], a["H"], a["D"], a["fs"],
                                    a["cs"], a["out"], None)

    assert call(D=96) == cslib.CS_ERR_UNSUPPORTED
    assert call(fs=128) == cslib.CS_ERR_INVALID_ARG
    assert call(out=None) == cslib.CS_ERR_INVALID_ARG
    assert call(fs=260) == cslib.CS_ERR_INVALID_ARG         # 520-byte rows break 16 B alignment
    assert call(H=17) == cslib.CS_ERR_UNSUPPORTED
    assert call(n=0, f=None, c=None, out=None) == cslib.CS_OK
    assert call() == cslib.CS_ERR_INVALID_ARG              # score_out over the key rows
    assert "overlaps" in cslib.cs_last_error_detail()


def test_select_rejects_bad_arguments(cslib):
    L = cslib.lib()
    assert L.cs_select_topk(FAKE, 10, 11, 0, FAKE, None) == cslib.CS_ERR_INVALID_ARG
    assert L.cs_select_topk(FAKE, 10, -1, 0, FAKE, None) == cslib.CS_ERR_INVALID_ARG
    assert L.cs_select_topk(FAKE, 10, 3, 0x7FFFFFFF - 5, FAKE, None) == cslib.CS_ERR_INVALID_ARG
    assert L.cs_select_topk(FAKE, 10, 3, -1, FAKE, None) == cslib.CS_ERR_INVALID_ARG
    assert L.cs_select_topk(None, 10, 3, 0, FAKE, None) == cslib.CS_ERR_INVALID_ARG
    assert L.cs_select_topk(None, 10, 0, 0, None, None) == cslib.CS_OK
    assert L.cs_select_topk(FAKE, 10, 3, 0, FAKE + 16, None) == cslib.CS_ERR_INVALID_ARG
    assert "overlaps" in cslib.cs_last_error_detail()


def test_attention_rejects_bad_arguments(cslib):
    L = cslib.lib()

    def call(**kw):
        a = dict(q=FAKE, k=FAKE, v=FAKE, o=FAKE, lse=None, dt=1, L=2, M=3, T=10, Hq=16, Hkv=2,
                 D=128, st=10 * 2 * 128, qpos=FAKE, scale=0.0884)
        a.update(kw)
        return L.cs_repair_attention(a["q"], a["k"], a["v"], a["o"], a["lse"], a["dt"], a["L"],
                                     a["M"], a["T"], a["Hq"], a["Hkv"], a["D"], a["st"],
                                     a["qpos"], a["scale"], None)

    assert call(Hq=15) == cslib.CS_ERR_INVALID_ARG
    assert call(D=64) == cslib.CS_ERR_UNSUPPORTED
    assert call(st=100) == cslib.CS_ERR_INVALID_ARG
    assert call(scale=float("nan")) == cslib.CS_ERR_INVALID_ARG
    assert call(T=0, st=0) == cslib.CS_ERR_INVALID_ARG
    assert call(qpos=None) == cslib.CS_ERR_INVALID_ARG
    assert call(o=FAKE + 4) == cslib.CS_ERR_INVALID_ARG
    assert call() == cslib.CS_ERR_INVALID_ARG           # o over k and v
    assert "overlaps" in cslib.cs_last_error_detail()
    assert call(Hq=256, Hkv=1) == cslib.CS_ERR_UNSUPPORTED
    assert call(M=0, q=None, o=None) == cslib.CS_OK
    # the optional LSE: 4-byte aligned, and not over k, v (read by other CTAs) or o
    far = FAKE + (1 << 24)
    assert call(o=far, lse=far + (1 << 20) + 2) == cslib.CS_ERR_INVALID_ARG
    assert "aligned" in cslib.cs_last_error_detail()
    assert call(o=far, lse=FAKE + 64) == cslib.CS_ERR_INVALID_ARG
    assert "lse overlaps k or v" in cslib.cs_last_error_detail()
    assert call(o=far, lse=far + 256) == cslib.CS_ERR_INVALID_ARG
    assert "lse overlaps o" in cslib.cs_last_error_detail()
    # query positions are read while other CTAs write o and lse
    assert call(o=far, qpos=far + 64) == cslib.CS_ERR_INVALID_ARG
    assert "qpos overlaps o" in cslib.cs_last_error_detail()
    assert call(o=far, lse=far + (1 << 20), qpos=far + (1 << 20) + 8) == cslib.CS_ERR_INVALID_ARG
    assert "qpos overlaps lse" in cslib.cs_last_error_detail()


def test_debug_wait_rejects_bad_limits(cslib):
    L = cslib.lib()
    assert L.cs_debug_wait_timeout(0, None) == cslib.CS_ERR_INVALID_ARG
    assert L.cs_debug_wait_timeout(20_000_000, None) == cslib.CS_ERR_INVALID_ARG


def test_python_binding_refuses_cpu_tensors(cslib):
    import torch
    k = torch.zeros(1, 4, 2, 128, dtype=torch.bfloat16)
    pos = torch.zeros(4, 3, dtype=torch.int32)
    with pytest.raises(ValueError):
        cslib.cs_rebase_keys(k, pos, pos)


def test_scatter_rejects_bad_arguments(cslib):
    L = cslib.lib()

    def call(**kw):
        a = dict(cache=FAKE, rows=FAKE + (1 << 24), dt=1, L=2, T=10, cst=10 * 256, n=3, rst=3 * 256,
                 re=256, idx=FAKE)
        a.update(kw)
        return L.cs_scatter_rows(a["cache"], a["rows"], a["dt"], a["L"], a["T"], a["cst"], a["n"],
                                 a["rst"], a["re"], a["idx"], None)

    assert call(dt=7) == cslib.CS_ERR_INVALID_ARG
    assert call(n=-1) == cslib.CS_ERR_INVALID_ARG
    assert call(re=0) == cslib.CS_ERR_INVALID_ARG
    assert call(re=5) == cslib.CS_ERR_UNSUPPORTED            # 10-byte rows
    assert call(cst=100) == cslib.CS_ERR_INVALID_ARG         # stride < T * row
    assert call(rst=100) == cslib.CS_ERR_INVALID_ARG
    assert call(idx=None) == cslib.CS_ERR_INVALID_ARG
    assert call(cache=FAKE + 8) == cslib.CS_ERR_INVALID_ARG  # misaligned
    assert call(rows=FAKE + 512) == cslib.CS_ERR_INVALID_ARG  # overlaps the cache
    assert call(idx=FAKE + 64) == cslib.CS_ERR_INVALID_ARG   # indices inside the cache
    assert "idx overlaps" in cslib.cs_last_error_detail()
    assert call(T=0, cst=0) == cslib.CS_ERR_INVALID_ARG
    assert call(n=0, rows=None, idx=None) == cslib.CS_OK
    assert call(L=0) == cslib.CS_OK


def test_rebase_and_score_rejects_bad_arguments(cslib):
    L = cslib.lib()
    r = cslib._RopeCfg(1e6, (ctypes.c_int32 * 3)(16, 24, 24))

    def call(**kw):
        a = dict(k_in=FAKE, k_out=FAKE, dt=1, L=2, stride=40 * 2 * 128, T=40, H=2, D=128, pl=FAKE,
                 pg=FAKE, sl=1, c0=8, nc=16, fr=FAKE + (1 << 24), fs=256, out=FAKE + (1 << 25))
        a.update(kw)
        return L.cs_rebase_and_score(a["k_in"], a["k_out"], a["dt"], a["L"], a["stride"], a["T"],
                                     a["H"], a["D"], a["pl"], a["pg"], ctypes.byref(r), a["sl"],
                                     a["c0"], a["nc"], a["fr"], a["fs"], a["out"], None)

    assert call(sl=2) == cslib.CS_ERR_INVALID_ARG           # score layer past the last
    assert call(sl=-1) == cslib.CS_ERR_INVALID_ARG
    assert call(c0=30) == cslib.CS_ERR_INVALID_ARG          # candidates past T
    assert call(nc=-1) == cslib.CS_ERR_INVALID_ARG
    assert call(fs=100) == cslib.CS_ERR_INVALID_ARG         # fresh rows shorter than a key row
    assert call(fr=FAKE + 8) == cslib.CS_ERR_INVALID_ARG    # misaligned fresh rows
    assert call(out=None) == cslib.CS_ERR_INVALID_ARG
    assert call(D=64) == cslib.CS_ERR_UNSUPPORTED
    assert call(out=FAKE + 64) == cslib.CS_ERR_INVALID_ARG  # score_out over the keys
    assert "overlaps" in cslib.cs_last_error_detail()
    assert call(fr=FAKE + 256) == cslib.CS_ERR_INVALID_ARG  # fresh rows inside the keys
    assert "overlaps" in cslib.cs_last_error_detail()
    far = FAKE + (1 << 26)
    assert call(pl=far, pg=far, out=far + 64) == cslib.CS_ERR_INVALID_ARG
    assert "coordinates overlap score_out" in cslib.cs_last_error_detail()
    assert call(L=0, nc=0) == cslib.CS_OK
