"""Checkpoint and resume of the decode loop.

The only state a sequence carries from one step to the next is its entropy
H_prev, temperature T and entropic time tau (Section 2, Section 3.3), plus
the caller's Philox seed and step offset; the sampler is counter-based, so a
loop restored from a checkpoint of those arrays must draw exactly the tokens
the uninterrupted loop draws.  The harness runs the closed loop of Section
3.4 on fixed per-step logits, writes the state to disk after step k, reloads
it in a fresh loop and compares every later token and state bit for bit.
It runs on the fp64 oracle on the CPU (which also checks the harness) and on
the CUDA path through the C ABI.
"""
import numpy as np
import pytest
import torch

import parity
import workloads

N_STEPS, K_SAVE, SEED = 6, 3, 77


def _logits_at(base, t):
    # a different distribution every step: the base rows shifted along V
    return torch.roll(base, shifts=7 * t + 1, dims=1).contiguous()


def _loop(run, lg0, start, stop, state):
    """Steps start..stop-1 of the closed loop; returns tokens and states per step."""
    dev = lg0["logits"].device
    T, H_prev, tau = (torch.from_numpy(np.asarray(state[k], np.float32)).to(dev)
                      for k in ("T", "H_prev", "tau"))
    toks, states = [], []
    for t in range(start, stop):
        lg = dict(lg0, logits=_logits_at(lg0["logits"], t), T_in=T, H_prev=H_prev, tau=tau)
        r = run(lg, SEED, t)
        assert (r["err"] == 0).all()
        st = {"T": np.asarray(r["T_out"], np.float32), "H_prev": np.asarray(r["H"], np.float32),
              "tau": np.asarray(r["tau"], np.float32)}
        toks.append(np.asarray(r["tok"]).copy())
        states.append(st)
        T, H_prev, tau = (torch.from_numpy(st[k]).to(dev) for k in ("T", "H_prev", "tau"))
    return toks, states


def _check_resume(run, lg0, tmp_path):
    init = {"T": lg0["T_in"].cpu().numpy(), "H_prev": lg0["H_prev"].cpu().numpy(),
            "tau": lg0["tau"].cpu().numpy()}
    toks, states = _loop(run, lg0, 0, N_STEPS, init)
    # checkpoint after step K_SAVE - 1: the three state arrays, the seed and
    # the next step's offset
    path = tmp_path / "ckpt.npz"
    np.savez(path, seed=SEED, offset=K_SAVE, **states[K_SAVE - 1])
    ck = np.load(path)
    assert int(ck["seed"]) == SEED
    toks2, states2 = _loop(run, lg0, int(ck["offset"]), N_STEPS,
                           {k: ck[k] for k in ("T", "H_prev", "tau")})
    for a, b in zip(toks[K_SAVE:], toks2):
        assert np.array_equal(a, b)
    for a, b in zip(states[K_SAVE:], states2):
        for k in a:
            assert np.array_equal(a[k], b[k]), k
    # the loop really moved: tokens and temperatures change across steps
    assert any(not np.array_equal(toks[0], x) for x in toks[1:])
    assert not np.array_equal(states[0]["T"], states[-1]["T"])
    # and restoring the wrong offset does not reproduce the draws: the same
    # logits and state at step K_SAVE, drawn with the next step's counter
    dev = lg0["logits"].device
    st = {k: torch.from_numpy(states[K_SAVE - 1][k]).to(dev) for k in ("T", "H_prev", "tau")}
    lg = dict(lg0, logits=_logits_at(lg0["logits"], K_SAVE), T_in=st["T"], H_prev=st["H_prev"],
              tau=st["tau"])
    assert np.array_equal(run(lg, SEED, K_SAVE)["tok"], toks[K_SAVE])
    assert not np.array_equal(run(lg, SEED, K_SAVE + 1)["tok"], toks[K_SAVE])
    return toks


def _workload():
    return workloads.WORKLOADS["llama3_8b"].scaled(B=24, V=4099)


def test_resume_on_the_oracle(oracle_lib, tmp_path):
    lg0 = workloads.make_logits(_workload(), "cpu")

    def run(lg, seed, t):
        return parity.oracle_ets(lg, seed=seed, offset=t)
    _check_resume(run, lg0, tmp_path)


@pytest.mark.gpu
def test_resume_on_the_gpu(tmp_path):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2603_03310_gb300 as eti
    eti.build()
    eti.load()
    lg0 = workloads.make_logits(_workload(), "cuda:0")

    def run(lg, seed, t):
        return parity.run_ets(eti, lg, seed=seed, offset=t)
    _check_resume(run, lg0, tmp_path)
