"""cure_tree_attn_noalloc on the GPU, against the oracle and cure_tree_attn.

The no-allocation entry point serves callers that cannot allocate device
memory (for example a plugin whose host framework owns all of HBM and hands
it only its inputs and outputs): it keeps the split-KV workspace in a fixed
64 MiB static device array instead of a caller buffer.  Its output must be the
tree attention the oracle computes, and the same as the workspace-taking
entry point's, call after call, even though every call reuses the array's
previous contents.

Its rejection of shapes beyond the array is checked on the host, with no GPU
reachable (tests/test_abi_host.py), so that a regression there can never
launch a kernel on buffers too small for the shape.

This file is collected last so that a failure here stops a `-x` run only
after every other test has run.
"""
import ctypes as C
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_00531_gb300 import workload as W

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda:0")
TOL = 2e-2            # the absolute tolerance of the attention parity tests
SCRATCH = 64 * 1024 * 1024
SCALE = 1.0 / math.sqrt(128)


@pytest.fixture(scope="module")
def env():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_00531_gb300 import _lib, cure
    torch.cuda.set_device(DEV)
    lib = _lib.load()
    P, I32 = C.c_void_p, C.c_int32
    lib.cure_tree_attn_noalloc.argtypes = [P, P, P, P, P, C.POINTER(_lib.KVDesc), P, P, P, I32, I32, I32,
                                           C.c_float, P, P]
    lib.cure_tree_attn_noalloc.restype = C.c_int
    return lib, cure


def _inputs(seed, B=4, K=16, budget=16, Hq=28, Hkv=4, lens=(0, 37, 1500, 4000)):
    rng = np.random.default_rng(seed)
    margin = (rng.integers(0, 8, size=(B, K)) * 0.25).astype(np.float32)
    ids = rng.integers(0, 1000, size=(B, K, 3))
    L = np.asarray(lens, dtype=np.int32)
    t = oracle.build_tree(ids, margin, rng.integers(0, 1000, size=B), L, 1.0, budget, 3, 1)
    N = 1 + K + budget
    table, npages = W.block_table(L, K, seed)
    q = W.normal_bf16((B, N, Hq, 128), 1.0, rng)
    tk = W.normal_bf16((B, N, Hkv, 128), 1.0, rng)
    tv = W.normal_bf16((B, N, Hkv, 128), 1.0, rng)
    kc = W.normal_bf16((npages, 16, Hkv, 128), 1.0, rng)
    vc = W.normal_bf16((npages, 16, Hkv, 128), 1.0, rng)
    return dict(t=t, q=q.to(DEV), tk=tk.to(DEV), tv=tv.to(DEV), kc=kc.to(DEV), vc=vc.to(DEV),
                host=dict(q=q, tk=tk, tv=tv, kc=kc, vc=vc), table_np=table,
                L=torch.from_numpy(L).to(DEV), L_np=L,
                table=torch.from_numpy(table).to(DEV), npages=npages, B=B, N=N, Hq=Hq, Hkv=Hkv,
                n=torch.from_numpy(t["n_nodes"].astype(np.int32)).to(DEV),
                anc=torch.from_numpy(t["anc"].view(np.int64)).to(DEV))


def _call_noalloc(lib, x, kv, out, in_place=False):
    s = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    tk, tv = (None, None) if in_place else (x["tk"].data_ptr(), x["tv"].data_ptr())
    return lib.cure_tree_attn_noalloc(
        x["q"].data_ptr(), tk, tv, x["kc"].data_ptr(), x["vc"].data_ptr(),
        C.byref(kv), x["L"].data_ptr(), x["n"].data_ptr(), x["anc"].data_ptr(), x["B"], x["N"], x["Hq"],
        SCALE, out.data_ptr(), s)


def _oracle(x, in_place=False):
    h = x["host"]
    f = W.bf16_to_f64
    tk, tv = (None, None) if in_place else (f(h["tk"]), f(h["tv"]))
    return oracle.tree_attn(f(h["q"]), tk, tv, f(h["kc"]), f(h["vc"]), x["L_np"], x["t"]["n_nodes"],
                            x["t"]["anc"], SCALE, x["table_np"], 16)


def _close(got, want):
    err = float((got - want).abs().max())
    return err <= TOL, err


def test_noalloc_matches_oracle_and_workspace_entry_point_on_two_calls(env):
    lib, cure = env
    for call, seed in enumerate((1, 2)):     # two calls in a row, different inputs
        x = _inputs(seed)
        kv = cure.kv_desc(x["Hkv"], 128, x["table"].shape[1], x["table"], 16, x["npages"])
        assert cure.cure_tree_attn_workspace_size(x["B"], x["N"], x["Hq"], kv) <= SCRATCH
        ref = cure.cure_tree_attn(x["q"], x["tk"], x["tv"], x["kc"], x["vc"], kv, x["L"], x["n"], x["anc"],
                                  SCALE)
        out = torch.full_like(ref, float("nan"))
        assert _call_noalloc(lib, x, kv, out) == 0
        torch.cuda.synchronize()
        assert cure.cure_device_error() == 0
        want = torch.from_numpy(_oracle(x))
        for b in range(x["B"]):
            nb = int(x["t"]["n_nodes"][b])
            got = out[b, :nb].float().cpu()
            assert torch.isfinite(got).all(), (call, b)
            ok, err = _close(got, want[b, :nb].float())
            assert ok, ("oracle", call, b, err)
            ok, err = _close(got, ref[b, :nb].float().cpu())
            assert ok, ("cure_tree_attn", call, b, err)


def test_noalloc_in_place_layout(env):
    """Both tree tensors NULL: the in-place layout (node j's rows at cache
    slot L + j), as in cure_tree_attn."""
    lib, cure = env
    x = _inputs(4)
    L = x["L_np"]
    table, npages = W.block_table(L, x["N"] - 1, 4)      # pages up to slot L + N - 1
    rng = np.random.default_rng(4)
    kc = W.normal_bf16((npages, 16, x["Hkv"], 128), 1.0, rng)
    vc = W.normal_bf16((npages, 16, x["Hkv"], 128), 1.0, rng)
    for b in range(x["B"]):
        for j in range(int(x["t"]["n_nodes"][b])):
            sl = int(L[b]) + j
            kc[int(table[b, sl // 16]), sl % 16] = x["host"]["tk"][b, j]
            vc[int(table[b, sl // 16]), sl % 16] = x["host"]["tv"][b, j]
    x = dict(x, kc=kc.to(DEV), vc=vc.to(DEV), table=torch.from_numpy(table).to(DEV), table_np=table,
             npages=npages, host=dict(x["host"], kc=kc, vc=vc))
    kv = cure.kv_desc(x["Hkv"], 128, table.shape[1], x["table"], 16, npages)
    ref = cure.cure_tree_attn(x["q"], None, None, x["kc"], x["vc"], kv, x["L"], x["n"], x["anc"], SCALE)
    out = torch.full_like(ref, float("nan"))
    assert _call_noalloc(lib, x, kv, out, in_place=True) == 0
    torch.cuda.synchronize()
    assert cure.cure_device_error() == 0
    want = torch.from_numpy(_oracle(x, in_place=True))
    for b in range(x["B"]):
        nb = int(x["t"]["n_nodes"][b])
        got = out[b, :nb].float().cpu()
        assert torch.isfinite(got).all(), b
        ok, err = _close(got, want[b, :nb].float())
        assert ok, ("oracle", b, err)
        ok, err = _close(got, ref[b, :nb].float().cpu())
        assert ok, ("cure_tree_attn", b, err)
