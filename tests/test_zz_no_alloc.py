"""af1_linear_forward_static, the forward entry point that allocates nothing
(its scratch is an array built into the library), against af1_linear_forward
on the same layer and input, twice in a row, through the C ABI, and both
against the FP64 oracle; af1_static_status then reports no timed-out wait.

Kept in a file of its own that sorts last, so that a run stopping at the
first failure has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

import synth
from oracle import af1_oracle as O
from tests.af1_cases import TOL, f16, signs_layer

pytestmark = pytest.mark.gpu


def test_static_scratch_entry_matches_workspace_entry():
    import paper_2609_06161_gb300 as P
    lib = P._lib
    fn = lib.af1_linear_forward_static
    fn.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p,
                   ctypes.c_int64, ctypes.c_int, ctypes.c_void_p]
    fn.restype = ctypes.c_int
    fwd = lib.af1_linear_forward
    stream = torch.cuda.current_stream().cuda_stream
    for (m, n, r, tokens) in [(1024, 4096, 800, 1), (4096, 4096, 2028, 5), (700, 900, 333, 17)]:
        d = synth.layer_signs(4242 + m + tokens, m, n, r, tokens)
        layer = signs_layer(P, d)
        x = f16(d["x"]).reshape(tokens, n)
        ldx = n + (-n) % 8
        if ldx != n:
            xp = torch.zeros((tokens, ldx), dtype=torch.float16, device="cuda")
            xp[:, :n] = x
            x = xp
        ldy = m + (-m) % 4
        ws = layer.make_workspace(tokens)
        oracle = O.forward_from_packed(O.pack_U(d["U"]), O.pack_V(d["V"]), d["a"], d["s"], d["b"], d["x"], m, n, r)
        y_ref = torch.empty((tokens, ldy), dtype=torch.float32, device="cuda")
        rc = fwd(layer._h, x.data_ptr(), ldx, tokens, y_ref.data_ptr(), ldy, 1, ws.data_ptr(),
                 ws.numel(), stream)
        assert rc == 0, P.last_error()
        for _ in range(2):
            y = torch.full((tokens, ldy), float("nan"), dtype=torch.float32, device="cuda")
            rc = fn(layer._h, x.data_ptr(), ldx, tokens, y.data_ptr(), ldy, 1, stream)
            assert rc == 0, P.last_error()
            torch.cuda.synchronize()
            a = y[:, :m].double().cpu().numpy()
            b = y_ref[:, :m].double().cpu().numpy()
            assert np.isfinite(a).all()
            assert O.rowwise_rel_err(a, b) <= TOL
            assert O.rowwise_rel_err(a, oracle) <= TOL
        P.static_status()  # raises AF1Error(AF1_ERR_TIMEOUT) if a wait of a static call gave up
        layer.free()


def test_static_scratch_rejects_oversized_layer():
    import paper_2609_06161_gb300 as P
    lib = P._lib
    fn = lib.af1_linear_forward_static
    fn.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p,
                   ctypes.c_int64, ctypes.c_int, ctypes.c_void_p]
    fn.restype = ctypes.c_int
    # r = 16384 needs 16 x 16384 floats of scratch plus a header: over 1 MiB.
    m, n, r = 64, 64, 16384
    g = synth.rng(1)
    Uw = torch.from_numpy(synth.random_words(g, m, 4 * ((r + 127) // 128), r).view(np.int32)).cuda()
    Vw = torch.from_numpy(synth.random_words(g, r, 4, n).view(np.int32)).cuda()
    a = f16(synth.scales_f16(g, m))
    s = f16(synth.scales_f16(g, r))
    b = f16(synth.scales_f16(g, n))
    layer = P.Layer.from_words(Uw, Vw, a, s, b, m, n, r, any_rank=True)
    x = torch.zeros((1, n), dtype=torch.float16, device="cuda")
    y = torch.zeros((1, m), dtype=torch.float16, device="cuda")
    rc = fn(layer._h, x.data_ptr(), n, 1, y.data_ptr(), m, 0, torch.cuda.current_stream().cuda_stream)
    assert rc == -8
    assert "scratch" in P.last_error()
    layer.free()
