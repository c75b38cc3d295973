"""The C-ABI library loads and exports every entry point that include/*.h declares,
and its host-side logic (validation, workspace sizing) behaves -- no GPU needed,
no kernel is launched."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
INCLUDE = os.path.join(ROOT, "include")


def _declared():
    names = set()
    for f in os.listdir(INCLUDE):
        if f.endswith(".h"):
            src = open(os.path.join(INCLUDE, f)).read()
            names |= set(re.findall(r"\b(moevie_\w+)\s*\(", src))
    return names


@pytest.fixture(scope="module")
def lib():
    from paper_2608_17402_gb300 import _build, moevie
    _build.build()
    return moevie.load()


def test_every_declared_symbol_is_exported(lib):
    declared = _declared()
    assert {"moevie_route", "moevie_permute", "moevie_expert_ffn", "moevie_combine",
            "moevie_moe_forward", "moevie_workspace_size"} <= declared
    for name in sorted(declared):
        assert hasattr(lib, name), name
    from paper_2608_17402_gb300 import moevie
    assert set(moevie.C_ENTRY_POINTS) == declared


def test_status_strings_and_version(lib):
    assert lib.moevie_status_string(0) == b"MOEVIE_OK"
    assert lib.moevie_status_string(3) == b"MOEVIE_ERR_WORKSPACE"
    assert lib.moevie_version() >= 100


def _ws_size(lib, *dims):
    out = ctypes.c_size_t(0)
    rc = lib.moevie_workspace_size(*dims, ctypes.byref(out))
    return rc, out.value


def test_workspace_size_monotone_and_validated(lib):
    rc, a = _ws_size(lib, 512, 768, 16, 2, 768, 0)
    assert rc == 0 and a > 0
    rc, b = _ws_size(lib, 1024, 768, 16, 2, 768, 0)
    assert rc == 0 and b > a
    rc, c = _ws_size(lib, 1024, 768, 16, 2, 768, 1024)
    assert rc == 0 and c > b
    assert _ws_size(lib, 512, 770, 16, 2, 768, 0)[0] == 2      # d % 8 != 0
    # any hidden width: rows of W1 and of the hidden activations are padded to 8 elements
    for h in (1, 13, 684, 760, 854):
        rc, w = _ws_size(lib, 512, 768, 16, 2, h, h)
        rc2, w2 = _ws_size(lib, 512, 768, 16, 2, h + 1, h + 1)
        assert rc == 0 and rc2 == 0 and w2 >= w, h
    assert _ws_size(lib, 512, 768, 16, 17, 768, 0)[0] == 2     # k > E
    assert _ws_size(lib, 512, 768, 2048, 2, 768, 0)[0] == 2    # E > 1024
    assert _ws_size(lib, -1, 768, 16, 2, 768, 0)[0] == 1
    assert lib.moevie_workspace_size(1, 8, 1, 1, 16, 0, None) == 1


def test_validation_happens_before_any_launch(lib):
    P = ctypes.c_void_p
    fake = P(0x1000)          # never dereferenced: every call below fails validation first
    # sizes outside the supported set
    assert lib.moevie_route(fake, fake, fake, 4, 12, 8, 2, fake, fake, fake, 1 << 20, None) == 2
    # null pointers with T > 0
    assert lib.moevie_route(None, fake, fake, 4, 16, 8, 2, fake, fake, fake, 1 << 20, None) == 1
    # misaligned x
    assert lib.moevie_route(P(0x1008), fake, fake, 4, 16, 8, 2, fake, fake, fake, 1 << 20, None) == 1
    # workspace too small
    assert lib.moevie_route(fake, fake, fake, 4, 16, 8, 2, fake, fake, fake, 16, None) == 3
    # T == 0 is a valid no-op
    assert lib.moevie_route(None, None, None, 0, 16, 8, 2, None, None, None, 0, None) == 0
    assert lib.moevie_moe_forward(None, fake, 4, fake, None, fake, 1 << 20, None) == 1
    assert lib.moevie_combine(fake, fake, fake, None, ctypes.c_float(1.0), 4, 2, 12, fake, None) == 2
    assert lib.moevie_test_wait_timeout(fake, 256, 0, None) == 1


def test_forward_rejects_bad_layer(lib):
    from paper_2608_17402_gb300.moevie import _Layer
    fake = 0x1000
    L = _Layer(16, 8, 2, 32, 0, fake, fake, fake, fake, 0, 0, 1.0)
    rc = lib.moevie_moe_forward(ctypes.byref(L), ctypes.c_void_p(fake), 4, ctypes.c_void_p(fake),
                                None, ctypes.c_void_p(fake), 16, None)
    assert rc == 3   # workspace too small
    L.k = 9          # k > E
    rc = lib.moevie_moe_forward(ctypes.byref(L), ctypes.c_void_p(fake), 4, ctypes.c_void_p(fake),
                                None, ctypes.c_void_p(fake), 1 << 30, None)
    assert rc == 2

    def fwd(layer, ws_bytes=1 << 30):
        return lib.moevie_moe_forward(ctypes.byref(layer), ctypes.c_void_p(fake), 4,
                                      ctypes.c_void_p(fake), None, ctypes.c_void_p(fake), ws_bytes, None)
    # every case below fails argument validation, before the workspace size check
    # and before anything is enqueued
    assert fwd(_Layer(16, 8, 2, 32, 32, fake, fake, fake, fake, fake, 0, 1.0)) == 1      # shared, no Ws2
    assert fwd(_Layer(16, 8, 2, 32, 32, fake, fake, fake, fake, fake, fake, 1.0,
                      fake, 0)) == 1                                                     # SwiGLU shared, no Ws3
    assert fwd(_Layer(16, 8, 2, 32, 0, fake, fake, fake, fake, 0, 0, 1.0, fake + 8)) == 1   # misaligned W3
    assert fwd(_Layer(16, 8, 2, 32, 0, fake, fake, fake + 4, fake, 0, 0, 1.0)) == 1          # misaligned W1
    # a hidden width that is not a multiple of 8 is supported: only the workspace is short
    assert fwd(_Layer(16, 8, 2, 13, 13, fake, fake, fake, fake, fake, fake, 1.0), 16) == 3


def test_shared_groups_plan_and_monotone_workspace(lib):
    """moevie_shared_groups: the shared expert rides in the routed GEMMs as h_s / h
    always-on groups when h divides h_s and the down-projection is not band-ordered
    (fp32 accumulator [T, d] <= 64 MiB); the workspace size stays monotone in T across
    that switch."""
    g = lib.moevie_shared_groups
    g.argtypes = [ctypes.c_int64] * 6
    g.restype = ctypes.c_int64
    assert g(8192, 1024, 64, 8, 512, 1024) == 2
    assert g(300, 128, 16, 4, 128, 384) == 3
    assert g(300, 256, 16, 4, 416, 128) == 0          # h does not divide h_s
    assert g(8192, 1024, 64, 8, 512, 0) == 0          # no shared expert
    assert g(65536, 1664, 256, 8, 416, 832) == 0      # band-ordered down-projection
    assert g(8192, 1023, 64, 8, 512, 1024) == 0       # invalid sizes
    assert g(8192, 768, 31, 3, 512, 512) == 1         # the paper's B model: one shared expert
    assert g(8192, 1024, 31, 3, 684, 684) == 1        # one chunk of a width that is not a multiple of 8
    assert g(8192, 1024, 31, 3, 684, 1368) == 0       # chunk 1 would start off a 16-byte boundary
    d = 1024
    t_switch = (64 << 20) // (4 * d)                  # accumulator reaches 64 MiB
    assert g(t_switch, d, 64, 8, 512, 1024) == 2 and g(t_switch + 1, d, 64, 8, 512, 1024) == 0
    prev = 0
    for T in range(t_switch - 4, t_switch + 5):
        rc, size = _ws_size(lib, T, d, 64, 8, 512, 1024)
        assert rc == 0 and size >= prev, T
        prev = size


def test_bias_update_validates_before_launch(lib):
    f = lib.moevie_update_bias
    f.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_float, ctypes.c_int, ctypes.c_void_p,
                  ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]
    p = ctypes.c_void_p(256)
    assert f(p, 0, 0.1, 0, p, p, 4096, None) == 1        # E < 1
    assert f(p, 1025, 0.1, 0, p, p, 4096, None) == 1     # E > 1024
    assert f(p, 8, 0.1, 2, p, p, 4096, None) == 1        # unknown rule
    assert f(None, 8, 0.1, 0, p, p, 4096, None) == 1     # null counts
    assert f(p, 8, 0.1, 0, p, p, 128, None) == 3         # workspace too small


def test_row_padding_helpers():
    """W1, W3, Ws1, Ws3 and the hidden activations have rows h rounded up to 8 elements
    apart: moevie_pad_rows lays a tensor out that way (a view of [..., h]) and returns a
    tensor that already is one unchanged; any other strides are rejected."""
    import torch
    from paper_2608_17402_gb300 import moevie
    assert [moevie.row_ld(h) for h in (1, 7, 8, 13, 512, 684, 854)] == [8, 8, 8, 16, 512, 688, 856]
    for shape in [(3, 5, 684), (5, 854), (2, 4, 13), (1, 3, 1)]:
        w = torch.randn(*shape)
        p = moevie.moevie_pad_rows(w)
        assert p.shape == w.shape and torch.equal(p, w) and moevie._rows_ok(p)
        assert p.stride()[-2] == moevie.row_ld(shape[-1])
        assert not moevie._rows_ok(w.contiguous())   # dense rows of a width that is not a multiple of 8
    w = torch.randn(4, 6, 512)
    assert moevie.moevie_pad_rows(w) is w
    with pytest.raises(ValueError):   # a host tensor is never accepted as device weights
        moevie._want_rows(w, torch.float32, "W1")


@pytest.mark.parametrize("d,E,k,h,hs", [(1024, 64, 8, 512, 1024), (768, 31, 3, 512, 512),
                                        (1024, 31, 3, 684, 684), (1280, 31, 7, 854, 854),
                                        (1664, 256, 8, 416, 0), (64, 4, 2, 13, 5), (96, 1, 1, 1, 0)])
def test_workspace_size_monotone_and_covers_the_big_regions(lib, d, E, k, h, hs):
    """For every T the workspace is monotone in T and at least holds the fp32 y
    accumulator [T, d] and the hidden activations [T k, h rounded up to 8] bf16."""
    hp = (h + 7) // 8 * 8
    prev = 0
    for T in list(range(0, 600, 37)) + [4095, 4096, 4097, 8192, 16383, 16384, 16385, 65536]:
        rc, size = _ws_size(lib, T, d, E, k, h, hs)
        assert rc == 0 and size >= prev, (T, size, prev)
        assert size >= 4 * T * d + 2 * T * k * hp
        prev = size


def test_backward_workspace_and_validation(lib):
    """moevie_backward_workspace_size grows with the shared expert's width and with SwiGLU,
    and moevie_moe_backward validates its layer and gradient pointers before any launch."""
    from paper_2608_17402_gb300.moevie import _Layer

    def size(*dims):
        out = ctypes.c_size_t(0)
        rc = lib.moevie_backward_workspace_size(*dims, ctypes.byref(out))
        return rc, out.value
    rc0, a = size(1024, 256, 16, 4, 128, 0, 0)
    rc1, b = size(1024, 256, 16, 4, 128, 256, 0)
    rc2, c = size(1024, 256, 16, 4, 128, 256, 1)
    assert rc0 == rc1 == rc2 == 0 and a < b < c
    assert size(2048, 256, 16, 4, 128, 256, 1)[1] > c          # monotone in T
    assert size(1024, 256, 16, 4, 128, 70000, 0)[0] == 2       # h_s above 65535
    assert size(1024, 256, 40, 33, 128, 0, 0)[0] == 2          # k above 32
    fake = 0x1000
    P = ctypes.c_void_p

    def bwd(layer, dWs1=fake, dWs2=fake, dWs3=None, ws_bytes=1 << 30):
        g = [P(fake)] * 5   # dx, dW_r, dW1, dW2 and (SwiGLU) dW3
        return lib.moevie_moe_backward(ctypes.byref(layer), P(fake), P(fake), 4, P(fake), g[0], g[1], g[2], g[3],
                                       None if layer.W3 == 0 else g[4], None if dWs1 is None else P(dWs1),
                                       None if dWs2 is None else P(dWs2), None if dWs3 is None else P(dWs3),
                                       P(fake), ws_bytes, None)
    shared = _Layer(16, 8, 2, 32, 32, fake, fake, fake, fake, fake, fake, 1.0)
    assert bwd(shared, ws_bytes=16) == 3                        # workspace too small
    assert bwd(shared, dWs1=None) == 1                          # shared expert without dWs1
    assert bwd(shared, dWs2=fake + 4) == 1                      # misaligned dWs2
    swiglu = _Layer(16, 8, 2, 32, 32, fake, fake, fake, fake, fake, fake, 1.0, fake, fake)
    assert bwd(swiglu) == 1                                     # SwiGLU shared expert without dWs3
    assert bwd(_Layer(16, 8, 2, 32, 32, fake, fake, fake, fake, fake, fake, 1.0, fake, 0), dWs3=fake) == 1


def test_forward_host_validation(lib):
    """moevie_moe_forward_host checks the chunk count, its buffers and the workspace (sized
    for one chunk) before creating its streams or enqueueing anything."""
    from paper_2608_17402_gb300 import moevie
    from paper_2608_17402_gb300.moevie import _Layer
    fake = 0x1000
    P = ctypes.c_void_p
    L = _Layer(16, 8, 2, 32, 0, fake, fake, fake, fake, 0, 0, 1.0)

    def fwd(T, chunks, ws_bytes, x_dev=fake, x_host=fake):
        return lib.moevie_moe_forward_host(ctypes.byref(L), None if x_host is None else P(x_host), T, P(fake),
                                           P(x_dev), P(fake), chunks, P(fake), ws_bytes, None)
    assert fwd(64, 0, 1 << 30) == 2
    assert fwd(64, moevie.HOST_MAX_CHUNKS + 1, 1 << 30) == 2
    assert fwd(64, 4, 1 << 30, x_dev=fake + 8) == 1             # misaligned device buffer
    assert fwd(64, 4, 1 << 30, x_host=None) == 1
    assert fwd(0, 4, 0) == 0                                    # T == 0: nothing to do
    out = ctypes.c_size_t(0)
    assert lib.moevie_workspace_size(16, 16, 8, 2, 32, 0, ctypes.byref(out)) == 0
    assert fwd(64, 2, out.value) == 3                           # chunks of 32 tokens need more room
    assert [moevie.host_chunks(T) for T in (1024, 8192, 16384, 32768, 65536, 1 << 20)] == [1, 1, 1, 2, 2, 16]


def test_header_is_plain_c(lib, tmp_path):
    """include/*.h compile as C11 (no C++ in the ABI), and a C program links against the
    library and calls a host-only entry point."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "abi.c"
    src.write_text(
        '#include <stdio.h>\n#include "moevie.h"\n#include "moevie_testing.h"\n'
        "int main(void) {\n"
        "    size_t bytes = 0;\n"
        "    moevie_layer layer = {0};\n"
        "    moevie_status s = moevie_workspace_size(512, 768, 16, 2, 768, 0, &bytes);\n"
        "    (void)layer;\n"
        '    printf("%d %zu\\n", (int)s, bytes);\n'
        "    return s;\n"
        "}\n")
    libdir = os.path.dirname(lib._name)
    exe = tmp_path / "abi"
    subprocess.run([gcc, "-std=c11", "-Wall", "-Wextra", "-Werror", "-I", INCLUDE, str(src), "-o", str(exe),
                    "-L", libdir, "-lmoevie", "-Wl,--unresolved-symbols=ignore-in-shared-libs",
                    f"-Wl,-rpath,{libdir}"], check=True, capture_output=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()
    rc, want = _ws_size(lib, 512, 768, 16, 2, 768, 0)
    assert out == ["0", str(want)] and rc == 0
