"""Helpers shared by the GPU parity tests: seeded layers in torch form, the
oracle's answer for them, and the tolerance (row-wise infinity-norm relative
error <= 2e-3 against the FP64 oracle, FP16 inputs, FP32 accumulation)."""
import numpy as np
import torch

import synth
from oracle import af1_oracle as O

TOL = 2e-3


def f16(bits, device="cuda"):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.float16)).to(device)


def signs_layer(P, d, any_rank=True, return_words=False, tc_decode=False, stream_decode=False, mma_decode=False,
                lut_decode=False):
    U = torch.from_numpy(d["U"]).cuda()
    V = torch.from_numpy(d["V"]).cuda()
    return P.Layer.from_signs(U, V, f16(d["a"]), f16(d["s"]), f16(d["b"]), any_rank=any_rank,
                              return_words=return_words, tc_decode=tc_decode, stream_decode=stream_decode,
                              mma_decode=mma_decode, lut_decode=lut_decode)


def words_layer(P, d, m, n, r, any_rank=True, tc_decode=False, stream_decode=False, mma_decode=False,
                lut_decode=False):
    Uw = torch.from_numpy(d["Uw"].view(np.int32)).cuda()
    Vw = torch.from_numpy(d["Vw"].view(np.int32)).cuda()
    return P.Layer.from_words(Uw, Vw, f16(d["a"]), f16(d["s"]), f16(d["b"]), m, n, r, any_rank=any_rank,
                              tc_decode=tc_decode, stream_decode=stream_decode, mma_decode=mma_decode,
                              lut_decode=lut_decode)


def oracle_from_signs(d, n, rows=None):
    m, r = d["U"].shape
    Uw, Vw = O.pack_U(d["U"]), O.pack_V(d["V"])
    return O.forward_from_packed(Uw, Vw, d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)


def run_gpu(layer, x_bits, n, out_dtype=torch.float32):
    x = f16(x_bits).reshape(-1, n)
    y = layer.forward(x, out_dtype=out_dtype)
    torch.cuda.synchronize()
    return y.double().cpu().numpy()
