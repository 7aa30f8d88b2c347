"""Failure detection on the GPU without a GPU fault.

* A grid barrier of the fused preparation kernel is made to wait for an
  arrival count that never comes (host-side injection): every block gives up
  after about a second, the device status records a timeout, the next call
  reports MOECA_ERR_TIMEOUT, and moeca_reset brings the handle back to
  results identical to a fresh handle's.
* A device allocation that cannot succeed is reported as MOECA_ERR_OOM and
  leaves nothing behind: a normal handle can be created right after.
* A cached expert id out of range, written by the host, is reported as a
  device status and cleared by moeca_reset.
"""
import ctypes

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def M():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2606_15615_gb300 import moeca
    return moeca


def _stack(M, seed=3):
    import torch
    from paper_2606_15615_gb300.workloads import tiny_layer
    T, D, E, k, F = 256, 128, 8, 2, 192
    w, x0, rng = tiny_layer(seed, T, D, E, k, F, n_shared=0, bias=False, wscale=0.05)
    cfg = M.moeca_config_default(n_layers=1, hidden=D, ffn=F, n_experts=E, top_k=k, max_tokens=T,
                                 dtype=M.MOECA_BF16, tau0=0.75)
    xs = [x0]
    for _ in range(2):
        xs.append((xs[-1] + 0.05 * rng.standard_normal(x0.shape)).astype(np.float32))
    dev = torch.device("cuda", 0)
    xs = [torch.from_numpy(x).to(dev).to(torch.bfloat16) for x in xs]
    return cfg, w, xs


def _run(st, xs):
    import torch
    outs = [st.step(x, t).clone() for t, x in enumerate(xs)]
    torch.cuda.synchronize()
    return outs


def test_barrier_stall_times_out_and_reset_recovers(M):
    import torch
    cfg, w, xs = _stack(M)
    ref = M.Stack(cfg, [w])
    expected = _run(ref, xs)
    ref.close()

    st = M.Stack(cfg, [w])
    st.step(xs[0], 0)
    M.moeca_inject_fault(st.handle, M.MOECA_FAULT_BARRIER_STALL)
    st.step(xs[1], 1)          # its barriers give up after about a second each
    torch.cuda.synchronize()
    with pytest.raises(M.MoecaError) as err:
        st.stats()
    assert err.value.status == M.MOECA_ERR_TIMEOUT
    with pytest.raises(M.MoecaError) as err:
        st.step(xs[2], 2)      # refused until the handle is reset
    assert err.value.status == M.MOECA_ERR_TIMEOUT

    M.moeca_reset(st.handle)
    st.stats()                 # the status is clear again
    got = _run(st, xs)
    for a, b in zip(got, expected):
        assert torch.equal(a, b)
    st.close()


def test_unsatisfiable_allocation_is_reported_and_leaves_nothing(M):
    import torch
    dev = torch.device("cuda", 0)
    dummy = torch.zeros(1024, dtype=torch.bfloat16, device=dev)
    cfg = M.moeca_config_default(n_layers=1, hidden=4096, ffn=16384, n_experts=4, top_k=2,
                                 max_tokens=1 << 24, dtype=M.MOECA_BF16)
    lw = M.moeca_layer_weights(w_gate=dummy.data_ptr(), b_gate=None, w1=dummy.data_ptr(),
                               w2=dummy.data_ptr(), ws1=None, ws2=None)
    h = ctypes.c_void_p()
    arr = (M.moeca_layer_weights * 1)(lw)
    free_before = torch.cuda.mem_get_info(dev)[0]
    assert M.LIB.moeca_create(ctypes.byref(cfg), arr, 0, ctypes.byref(h)) == M.MOECA_ERR_OOM
    assert b"device allocation" in M.LIB.moeca_last_error(None)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info(dev)[0] >= free_before - (64 << 20)
    cfg2, w, xs = _stack(M)
    st = M.Stack(cfg2, [w])
    _run(st, xs[:1])
    st.close()


def test_corrupted_cache_metadata_is_reported(M):
    """A cached expert id out of range, written by the host through
    moeca_set_layer_state, is reported as MOECA_ERR_DEVICE_STATUS; the branch
    is treated as unmatched, and moeca_reset clears the status."""
    import torch
    cfg, w, xs = _stack(M, seed=5)
    st = M.Stack(cfg, [w])
    st.step(xs[0], 0)
    state = st.get_state(0)
    torch.cuda.synchronize()
    bad = {k_: (v.clone() if isinstance(v, torch.Tensor) else v) for k_, v in state.items()}
    bad["cache_e"][5, 0] = 999
    st.set_state(0, bad)
    st.step(xs[1], 1)
    torch.cuda.synchronize()
    with pytest.raises(M.MoecaError) as err:
        st.stats()
    assert err.value.status == M.MOECA_ERR_DEVICE_STATUS
    M.moeca_reset(st.handle)
    _run(st, xs)
    st.stats()
    st.close()
