"""The no-allocation sampling entry point agrees with the regular one.

eti_entropy_temp_sample_noalloc serves callers that cannot allocate device
memory (a plugin handed only its input and output buffers, a latency-critical
thread that must stay out of the allocator): it keeps its scratch in a fixed
array inside the library instead of a caller workspace.  These checks call it
through the C ABI, twice in a row (the second call finds the first call's
leftovers in the shared array), and compare every output with
eti_entropy_temp_sample on the same inputs, within the parity tolerances.
This file is collected last and builds and loads the library itself, so it
runs the same alone in a fresh process or after the other tests.
"""
import math

import numpy as np
import pytest
import torch

import parity
import workloads

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module")
def eti():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2603_03310_gb300 as m
    m.build()
    m.load()
    return m


def _outputs(B, dev):
    f32, i32 = torch.float32, torch.int32
    return dict(tok=torch.full((B,), -7, dtype=i32, device=dev),
                H=torch.full((B,), -7.0, dtype=f32, device=dev),
                T_out=torch.full((B,), -7.0, dtype=f32, device=dev),
                dH=torch.full((B,), -7.0, dtype=f32, device=dev),
                theta_next=torch.full((B,), -7.0, dtype=f32, device=dev),
                surprisal=torch.full((B,), -7.0, dtype=f32, device=dev),
                err=torch.full((B,), -7, dtype=i32, device=dev))


def _call(eti, fn, lg, seed, offset, with_ws):
    B = lg["logits"].shape[0]
    o = _outputs(B, lg["logits"].device)
    tau = lg["tau"].clone()
    kw = dict(seed=seed, offset=offset, dH=o["dH"], theta_next=o["theta_next"],
              tok_surprisal=o["surprisal"])
    args = (lg["logits"], lg["T_in"], lg["H_prev"], tau, lg["H_target"], o["tok"], o["H"],
            o["T_out"], o["err"])
    if with_ws:
        ws = torch.empty(eti.entropy_temp_sample_workspace_size(B, lg["logits"].shape[1]),
                         dtype=torch.uint8, device=lg["logits"].device)
        fn(*args, ws, **kw)
    else:
        fn(*args, **kw)
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in o.items()}
    res["tau"] = tau.cpu().numpy()
    res["err"] = res["err"].view(np.uint32)
    return res


def _agree(a, b):
    """Same error bits and tokens; every float within the parity tolerances."""
    assert np.array_equal(a["err"], b["err"])
    assert np.array_equal(a["tok"], b["tok"])
    ok = a["err"] == 0
    for k, rel, abs_ in (("H", parity.H_REL, parity.H_ABS_SMALL), ("T_out", 1e-4, 0.0),
                         ("dH", 1e-4, 1e-5), ("tau", 1e-4, 1e-5), ("theta_next", 0.0, 2e-4),
                         ("surprisal", 1e-4, 1e-5)):
        x, y = a[k][ok].astype(np.float64), b[k][ok].astype(np.float64)
        assert np.all(np.abs(x - y) <= np.maximum(rel * np.abs(y), abs_)), k


def test_noalloc_matches_workspace_entry_point_twice(eti):
    # two different problems back to back: the second call runs on the
    # scratch contents the first one left behind
    cases = [(workloads.WORKLOADS["llama3_8b"], 11, 3), (workloads.WORKLOADS["tiny"], 0, 0)]
    for w, seed, offset in cases:
        lg = workloads.make_logits(w, DEV)
        ref = _call(eti, eti.eti_entropy_temp_sample, lg, seed, offset, with_ws=True)
        got = _call(eti, eti.eti_entropy_temp_sample_noalloc, lg, seed, offset, with_ws=False)
        _agree(got, ref)
        assert (got["err"] == 0).all() and (got["tok"] >= 0).all()
    # the same problem twice in a row gives the same answer
    w = workloads.WORKLOADS["mixed_batch"].scaled(B=48)
    lg = workloads.make_logits(w, DEV)
    first = _call(eti, eti.eti_entropy_temp_sample_noalloc, lg, 4, 9, with_ws=False)
    second = _call(eti, eti.eti_entropy_temp_sample_noalloc, lg, 4, 9, with_ws=False)
    _agree(second, first)
    _agree(second, _call(eti, eti.eti_entropy_temp_sample, lg, 4, 9, with_ws=True))


def test_noalloc_rejects_problems_beyond_its_scratch(eti):
    lib = eti.load()
    cap = lib.eti_entropy_temp_sample_noalloc_max_bytes()
    assert cap >= 64 * 1024
    # find the smallest batch that no longer fits; the call must refuse it
    # before touching any buffer (all pointers below are never dereferenced)
    B = 1
    while lib.eti_entropy_temp_sample_workspace_size(B, 4) <= cap:
        B *= 2
    assert B <= 65535
    x = torch.zeros(1, device=DEV)
    p = eti.ctrl_params()
    import ctypes
    ptr = ctypes.c_void_p(x.data_ptr())
    st = lib.eti_entropy_temp_sample_noalloc(ptr, B, 4, 4, ptr, ptr, ptr, ptr, ctypes.byref(p),
                                             0, 0, None, ptr, ptr, ptr, None, None, None, None, ptr,
                                             None)
    assert st == -7
    assert "fixed scratch" in lib.eti_status_string(st).decode()
