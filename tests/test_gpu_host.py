"""gmc_compress_host: the same call from and to page-locked host memory.

The host-buffer entry point copies the inputs itself (the hidden states on the
library's side stream, beside the kernels that do not read them) and copies
the outputs back.  Its outputs must be bit-identical to gmc_compress on the
same device inputs, on the pipelined path (one image; a ragged batch) and on
the identity path (K = N), and a second call reusing the buffers must see its
own inputs.
"""

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02134_gb300 import gmc
    gmc.lib()


def _host_inputs(wl):
    host = {}
    for k, v in wl.abi_arrays().items():
        if k == "text_offsets":
            continue
        t = torch.from_numpy(np.ascontiguousarray(v))
        if v.dtype == np.uint16:
            t = t.view(torch.int16).view(torch.bfloat16)
        host[k] = t.pin_memory()
    return host


def _run_both(wl, K=None):
    from paper_2608_02134_gb300 import gmc
    dt = gmc.GMC_BF16 if wl.dtype == "bf16" else gmc.GMC_F32
    comp = gmc.Compressor(wl.B, wl.gh, wl.gw, wl.T_max, wl.H, wl.Hkv, wl.d, wl.D,
                          wl.K if K is None else K, dt,
                          text_lengths=wl.T if wl.ragged else None)
    host = _host_inputs(wl)
    dev = {k: v.cuda() for k, v in host.items()}
    out = comp.run(dev["hidden"], dev["keys"], dev["queries"], dev["pos_ids"], dev["vo_probe"])
    torch.cuda.synchronize()
    ref = {k: t.clone() for k, t in (("idx", out.idx), ("hidden", out.hidden), ("kv", out.kv),
                                     ("pos", out.pos))}
    assert comp.status() == 0
    host_out = {k: torch.empty(v.shape, dtype=v.dtype).pin_memory() for k, v in ref.items()}
    dev_in = {k: torch.empty_like(v) for k, v in dev.items()}  # fresh device staging buffers
    comp.run_host(host, dev_in, host_out)
    torch.cuda.synchronize()
    assert comp.status() == 0
    return ref, host_out, comp, host, dev_in


def _same(ref, host_out):
    for k in ("idx", "hidden", "kv", "pos"):
        a = ref[k].cpu()
        b = host_out[k]
        if a.dtype == torch.bfloat16:
            a, b = a.view(torch.int16), b.view(torch.int16)
        assert torch.equal(a, b), f"{k} differs"


def test_host_call_matches_device_call_one_image():
    from paper_2608_02134_gb300 import workloads
    ref, host_out, comp, host, dev_in = _run_both(workloads.make("qwen"))
    _same(ref, host_out)
    # a second call reuses the device staging buffers: the outputs follow the
    # new host inputs, not leftovers of the first call
    host2 = {k: v.clone().pin_memory() for k, v in host.items()}
    host2["hidden"].copy_(torch.flip(host["hidden"], dims=[0]))
    out2 = {k: torch.empty_like(v).pin_memory() for k, v in host_out.items()}
    comp.run_host(host2, dev_in, out2)
    torch.cuda.synchronize()
    dev2 = {k: v.cuda() for k, v in host2.items()}
    o = comp.run(dev2["hidden"], dev2["keys"], dev2["queries"], dev2["pos_ids"], dev2["vo_probe"])
    torch.cuda.synchronize()
    _same({"idx": o.idx, "hidden": o.hidden, "kv": o.kv, "pos": o.pos}, out2)


def test_host_call_matches_device_call_ragged_batch():
    from paper_2608_02134_gb300 import workloads
    ref, host_out, *_ = _run_both(workloads.make("serving"))
    _same(ref, host_out)


def test_host_call_identity():
    from paper_2608_02134_gb300 import workloads
    wl = workloads.make("tiny")
    ref, host_out, *_ = _run_both(wl, K=wl.N)
    _same(ref, host_out)
    assert np.array_equal(host_out["idx"].numpy(), np.arange(wl.N, dtype=np.int32))
