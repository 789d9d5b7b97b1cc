"""twinkv_repair_host: the audit and swap (Sec. 3.4) on host-resident caches, in chunks
whose host<->device copies overlap the computation.  Its outputs must equal those of
twinkv_repair on the same inputs bit for bit (each unit is computed by the same kernels
on the same data), and the selection must equal the oracle's on the GPU's own b values
(split check).  Chunk sizes cover one unit, a ragged last chunk, the default and all
units; back-to-back calls check the ordering of successive calls' use of the arena."""
import numpy as np
import pytest
import torch

import oracle
from gpu_harness import device, keys_tensor, split_check
from paper_2608_27128_gb300 import synth
from paper_2608_27128_gb300 import twinkv as tk

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _setup():
    oracle.build()
    tk.load()
    torch.cuda.init()


def _case(name, L, H, N, ratio):
    w = synth.get(name, L=L, H=H, N=N)
    keys, _ = synth.keys(w)
    return w, keys, synth.masks(w, ratio)


def _host_keys(keys, L, H, pin):
    U, N, d = keys.shape
    if keys.dtype == np.float32:
        t = torch.from_numpy(keys.reshape(L, H, N, d).copy())
    else:
        t = torch.from_numpy(keys.view(np.int16).reshape(L, H, N, d).copy()).view(torch.bfloat16)
    return t.pin_memory() if pin else t


def _device_run(keys, S0, L, H, tau, want_all):
    U, N, _ = keys.shape
    out = tk.twinkv_repair(keys_tensor(keys, L, H),
                           torch.from_numpy(S0.reshape(L, H, N).copy()).to(device()),
                           torch.from_numpy(S0.sum(1).astype(np.int32)).to(device()),
                           threshold=tau, want_all=want_all)
    torch.cuda.synchronize()
    return {k: v.cpu() for k, v in out.items()}


def _host_run(keys, S0, L, H, tau, want_all, chunk, pin, stream=None):
    U, N, _ = keys.shape
    m = torch.from_numpy(S0.reshape(L, H, N).copy())
    b = torch.from_numpy(S0.sum(1).astype(np.int32))
    if pin:
        m, b = m.pin_memory(), b.pin_memory()
    return tk.twinkv_repair_host(_host_keys(keys, L, H, pin), m, b, threshold=tau,
                                 want_all=want_all, chunk_units=chunk, stream=stream)


def _assert_same(h, d):
    """Equal outputs; a unit's swap list is defined up to its nswaps entries only."""
    assert set(h) == set(d)
    for k in d:
        assert h[k].device.type == "cpu"
        if k != "swaps":
            assert torch.equal(h[k], d[k]), k
    for u, m in enumerate(d["nswaps"].tolist()):
        assert torch.equal(h["swaps"][u, :max(m, 0)], d["swaps"][u, :max(m, 0)]), u


@pytest.mark.parametrize("chunk,pin", [(0, True), (1, True), (4, True), (6, True),
                                       (100, False), (0, False)])
def test_host_path_equals_device_path(chunk, pin):
    L, H = 2, 3
    w, keys, S0 = _case("llama", L, H, 1500, 0.5)
    d = _device_run(keys, S0, L, H, w.tau, want_all=True)
    h = _host_run(keys, S0, L, H, w.tau, True, chunk, pin)
    torch.cuda.synchronize()
    _assert_same(h, d)
    hn = {k: v.numpy() for k, v in h.items()}
    split_check(hn, S0, w.tau, synth.N_SINK, synth.N_RECENT)
    assert np.all(hn["status"] == 0)


def test_host_path_pyramid_budgets():
    """Per-layer budgets: every chunk carries units of different |S0|."""
    L, H = 5, 2
    w = synth.get("qwen", L=L, H=H, N=1024)
    keys, _ = synth.keys(w)
    S0 = synth.masks(w, 0.5, schedule="pyramid")
    d = _device_run(keys, S0, L, H, w.tau, want_all=True)
    h = _host_run(keys, S0, L, H, w.tau, True, 3, True)
    torch.cuda.synchronize()
    _assert_same(h, d)
    hn = {k: v.numpy() for k, v in h.items()}
    split_check(hn, S0, w.tau, synth.N_SINK, synth.N_RECENT)
    np.testing.assert_array_equal(hn["mask"].reshape(L * H, -1).sum(1),
                                  np.repeat(synth.pyramid_budgets(w, 0.5), H))


def test_host_path_fp32_keys_and_no_scores():
    w, keys, S0 = _case("tiny", 1, 1, 512, 0.5)
    d = _device_run(keys, S0, 1, 1, w.tau, want_all=False)
    h = _host_run(keys, S0, 1, 1, w.tau, False, 0, True)
    torch.cuda.synchronize()
    _assert_same(h, d)


def test_back_to_back_calls_on_a_side_stream():
    """Two calls without a synchronisation between them share the binding's arena and
    the library's copy streams; each must still see its own inputs."""
    L, H = 1, 5
    w1, k1, m1 = _case("qwen", L, H, 2048, 0.3)
    k2 = synth.random_keys(5, L * H, 2048, 128)
    m2 = synth.random_masks(6, L * H, 2048, 700)
    d1 = _device_run(k1, m1, L, H, 0.85, True)
    d2 = _device_run(k2, m2, L, H, 0.3, True)
    st = torch.cuda.Stream()
    with torch.cuda.stream(st):
        h1 = _host_run(k1, m1, L, H, 0.85, True, 2, True, stream=st)
        h2 = _host_run(k2, m2, L, H, 0.3, True, 2, True, stream=st)
    st.synchronize()
    _assert_same(h1, d1)
    _assert_same(h2, d2)


def test_default_chunk_fills_whole_waves():
    """chunk_units = 0: about an eighth of the units, in whole waves of 128-row blocks
    over the SMs, and the arena size agrees with the explicit value."""
    import math
    sms = torch.cuda.get_device_properties(device()).multi_processor_count
    for L, H, N, d in [(36, 8, 16384, 128), (16, 8, 8192, 64), (1, 8, 131072, 128),
                       (2, 3, 1500, 64), (36, 8, 32768, 128)]:
        s = tk.Shape(L, H, N, d, tk.BF16)
        uc = tk.twinkv_host_default_chunk(s)
        U, rb = L * H, -(-N // 128)
        step = sms // math.gcd(sms, rb)
        assert 1 <= uc <= U
        if step <= U:
            assert uc % step == 0 and (uc * rb) % sms == 0
            assert abs(uc - (U + 7) // 8) <= step // 2 + 1 or uc == step
        assert tk.twinkv_host_arena_size(s, 0) == tk.twinkv_host_arena_size(s, uc)
    assert tk.twinkv_host_default_chunk(tk.Shape(0, 8, 100, 64, tk.BF16)) == 0


def test_arena_too_small_is_rejected():
    L, H = 1, 2
    _, keys, S0 = _case("llama", L, H, 600, 0.5)
    s = tk.Shape(L, H, 600, 64, tk.BF16)
    n = tk.twinkv_host_arena_size(s, 1)
    assert n > 0
    small = torch.empty(n - 256, dtype=torch.uint8, device=device())
    with pytest.raises(tk.TwinKVError) as e:
        tk.twinkv_repair_host(_host_keys(keys, L, H, False),
                              torch.from_numpy(S0.reshape(L, H, 600).copy()),
                              threshold=0.9, chunk_units=1, arena=small)
    assert e.value.status == tk.ERR_WORKSPACE
