"""phsa_step_host: the whole path for tensors in host memory.

Its kernels are the device-path calls' kernels on device copies of the same
inputs, so every result must be bit-identical to those calls (which the other
GPU tests hold against the oracle). Covered: both backward paths (two query
heads per KV head: tcgen05 kernels; one: CUDA cores), ragged lengths, calls
that alternate two workspaces with completion events (the copies of one call
overlap the kernels of the other), reuse of one workspace, outputs that are
not requested, and argument errors.
"""
import numpy as np
import pytest
import torch

from paper_2601_02819_gb300 import inputs, phsa

pytestmark = pytest.mark.gpu


def _workload(Hq, Hkv, L, topk, seed):
    return inputs.custom("host_step", B=2, L=L, Hq=Hq, Hkv=Hkv, topk=topk, n_init=1, n_local=2,
                         punct="sentence", seed=seed)


def _host_inputs(x):
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).pin_memory()
    return ({k: pin(x[k]) for k in ("Q", "K", "V", "dO")},
            torch.from_numpy(x["mask"]).pin_memory())


def _device_path(x, w):
    t = lambda a: torch.from_numpy(a.view(np.int16)).cuda().view(torch.bfloat16)
    Q, K, V, dO = t(x["Q"]), t(x["K"]), t(x["V"]), t(x["dO"])
    mask = torch.from_numpy(x["mask"]).cuda()
    Kr = phsa.phsa_build_block_repr(K, mask, w.lam)
    idx, cnt = phsa.phsa_select_blocks(Q, Kr, w.Hkv, w.topk, w.n_init, w.n_local, w.sm_scale)
    O, lse = phsa.phsa_sparse_attn_fwd(Q, K, V, idx, cnt, w.sm_scale)
    dQ, dK, dV = phsa.phsa_sparse_attn_bwd(Q, K, V, O, dO, lse, idx, cnt, w.sm_scale)
    torch.cuda.synchronize()
    bits = lambda a: a.view(torch.int16).cpu().numpy()
    return {"O": bits(O), "lse": lse.cpu().numpy(), "dQ": bits(dQ), "dK": bits(dK),
            "dV": bits(dV), "idx": idx.cpu().numpy(), "cnt": cnt.cpu().numpy()}


def _outputs(w):
    pinned = lambda shape, dt: torch.empty(shape, dtype=dt).pin_memory()
    NQB = -(-w.L // w.block_size)
    return {"O": pinned((w.B, w.Hq, w.L, w.D), torch.int16),
            "lse": pinned((w.B, w.Hq, w.L), torch.float32),
            "dQ": pinned((w.B, w.Hq, w.L, w.D), torch.int16),
            "dK": pinned((w.B, w.Hkv, w.L, w.D), torch.int16),
            "dV": pinned((w.B, w.Hkv, w.L, w.D), torch.int16),
            "idx": pinned((w.B, w.Hkv, NQB, w.topk), torch.int32),
            "cnt": pinned((w.B, w.Hkv, NQB), torch.int32)}


def _call(w, hin, hmask, out, ws, ev=None):
    phsa.phsa_step_host(hin["Q"], hin["K"], hin["V"], hin["dO"], hmask, w.lam, w.topk, w.n_init,
                        w.n_local, w.sm_scale, O=out["O"], lse=out["lse"], dQ=out["dQ"],
                        dK=out["dK"], dV=out["dV"], block_idx=out["idx"], block_cnt=out["cnt"],
                        workspace=ws, done_event=ev)


def _assert_equal(out, ref):
    for k, v in ref.items():
        got = out[k].numpy()
        assert np.array_equal(got, v), k


@pytest.mark.parametrize("Hq,Hkv", [(4, 2), (2, 2)])
def test_host_step_equals_device_path(Hq, Hkv):
    w = _workload(Hq, Hkv, 64 * 19 + 23, 6, seed=11)
    x = inputs.make_inputs(w, with_grad=True)
    hin, hmask = _host_inputs(x)
    ref = _device_path(x, w)
    out = _outputs(w)
    ws = torch.empty(phsa.phsa_step_host_workspace(w.B, w.L, w.Hq, w.Hkv, w.topk),
                     dtype=torch.uint8, device="cuda")
    _call(w, hin, hmask, out, ws)  # no event: the stream waits for the copies back
    torch.cuda.current_stream().synchronize()
    _assert_equal(out, ref)
    assert phsa.phsa_get_device_status() == 0
    phsa.phsa_step_host_release(ws)


def test_host_step_alternating_workspaces_overlap_and_stay_exact():
    w = _workload(4, 2, 64 * 33, 8, seed=0)
    xs = [inputs.make_inputs(w, with_grad=True, seed=100 + i) for i in range(4)]
    refs = [_device_path(x, w) for x in xs]
    hins = [_host_inputs(x) for x in xs]
    outs = [_outputs(w) for _ in xs]
    nbytes = phsa.phsa_step_host_workspace(w.B, w.L, w.Hq, w.Hkv, w.topk)
    wss = [torch.empty(nbytes, dtype=torch.uint8, device="cuda") for _ in range(2)]
    evs = [torch.cuda.Event() for _ in xs]
    # four steps on two workspaces: steps 2 and 3 reuse the workspaces of 0 and 1
    for i, (x, (hin, hmask)) in enumerate(zip(xs, hins)):
        _call(w, hin, hmask, outs[i], wss[i % 2], evs[i])
    for ev in evs:
        ev.synchronize()
    for out, ref in zip(outs, refs):
        _assert_equal(out, ref)
    assert phsa.phsa_get_device_status() == 0
    for ws in wss:
        phsa.phsa_step_host_release(ws)


def test_host_step_skips_outputs_not_requested_and_rejects_bad_arguments():
    w = _workload(4, 2, 64 * 6 + 5, 4, seed=3)
    x = inputs.make_inputs(w, with_grad=True)
    hin, hmask = _host_inputs(x)
    ref = _device_path(x, w)
    nbytes = phsa.phsa_step_host_workspace(w.B, w.L, w.Hq, w.Hkv, w.topk)
    ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    O, lse, dQ, dK, dV = phsa.phsa_step_host(hin["Q"], hin["K"], hin["V"], hin["dO"], hmask,
                                             w.lam, w.topk, w.n_init, w.n_local, w.sm_scale,
                                             workspace=ws)
    torch.cuda.current_stream().synchronize()
    assert np.array_equal(dK.view(torch.int16).numpy(), ref["dK"])
    assert np.array_equal(O.view(torch.int16).numpy(), ref["O"])
    with pytest.raises(phsa.PhsaError):  # one byte short
        phsa.phsa_step_host(hin["Q"], hin["K"], hin["V"], hin["dO"], hmask, w.lam, w.topk,
                            workspace=ws[: nbytes - 1])
    with pytest.raises(ValueError):  # device tensors are not host buffers
        phsa.phsa_step_host(hin["Q"].cuda(), hin["K"], hin["V"], hin["dO"], hmask, w.lam, w.topk,
                            workspace=ws)
    phsa.phsa_step_host_release(ws)
