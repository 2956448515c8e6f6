"""certkv_compress_host (host inputs, copies overlapped with the compression)
gives exactly what certkv_compress gives on the same data, for every chunk
size, with pinned and with pageable host memory; with a host output the
packed cache copied back chunk by chunk equals the device one."""
import pytest
import torch

from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu

WL = W.Workload("S", B=2, L=3, Hq=8, H=2, n=3000, d=128, w=20, keep=(1, 10), kind="planted")


def _reference(K, V, Q, B_live, params):
    return ck.certkv_compress(K, V, Q, B_live, params, with_tail=True)


def _same(a: ck.Packed, b: ck.Packed):
    assert torch.equal(a.real_counts, b.real_counts)
    assert torch.equal(a.offsets, b.offsets)
    n = int(a.offsets[-1])
    assert torch.equal(a.positions[:n], b.positions[:n])
    assert torch.equal(a.k[:n].view(torch.int16), b.k[:n].view(torch.int16))
    assert torch.equal(a.v[:n].view(torch.int16), b.v[:n].view(torch.int16))
    assert torch.equal(a.tail_f32, b.tail_f32)
    assert torch.equal(a.tail_mass, b.tail_mass)


@pytest.mark.parametrize("chunk", [1, 4, 0])
@pytest.mark.parametrize("pinned", [True, False])
def test_host_pipeline_equals_device_call(chunk, pinned):
    K, V, Q = W.draw(WL, device="cuda")
    params = ck.certkv_default_params()
    ref = _reference(K, V, Q, WL.B_live, params)
    hK, hV, hQ = K.cpu(), V.cpu(), Q.cpu()
    if pinned:
        hK, hV, hQ = hK.pin_memory(), hV.pin_memory(), hQ.pin_memory()
    got = ck.certkv_compress_host(hK, hV, hQ, WL.B_live, params, chunk=chunk, with_tail=True)
    torch.cuda.synchronize()
    _same(got, ref)


def test_host_pipeline_status_and_reuse():
    # two calls in a row on one workspace; the status word stays clean
    K, V, Q = W.draw(WL, device="cuda")
    params = ck.certkv_default_params()
    shape = ck.shape_of(K, Q)
    ws = ck.workspace(ck.certkv_host_workspace_bytes(shape, params, 2), K.device)
    hK, hV, hQ = K.cpu().pin_memory(), V.cpu().pin_memory(), Q.cpu().pin_memory()
    a = ck.certkv_compress_host(hK, hV, hQ, WL.B_live, params, chunk=2, ws=ws, with_tail=True)
    b = ck.certkv_compress_host(hK, hV, hQ, WL.B_live, params, chunk=2, ws=ws, with_tail=True)
    torch.cuda.synchronize()
    _same(a, b)
    assert ck.certkv_read_status(ws) == 0


@pytest.mark.parametrize("chunk", [1, 4, 0])
def test_host_copyback_equals_device_output(chunk):
    K, V, Q = W.draw(WL, device="cuda")
    params = ck.certkv_default_params()
    ref = _reference(K, V, Q, WL.B_live, params)
    hK, hV, hQ = K.cpu().pin_memory(), V.cpu().pin_memory(), Q.cpu().pin_memory()
    host = ck.Packed.empty_host(WL.B, WL.L, WL.H, WL.d, WL.B_live)
    for t in (host.k, host.v):
        t.view(torch.int16).fill_(-1)
    host.positions.fill_(-7)
    got = ck.certkv_compress_host(hK, hV, hQ, WL.B_live, params, chunk=chunk, with_tail=True,
                                  host_out=host)
    torch.cuda.synchronize()  # the copies back complete with the call's stream
    _same(got, ref)
    assert torch.equal(host.real_counts, ref.real_counts.cpu())
    assert torch.equal(host.offsets, ref.offsets.cpu())
    n = int(ref.offsets[-1])
    assert torch.equal(host.positions[:n], ref.positions[:n].cpu())
    assert torch.equal(host.k[:n].view(torch.int16), ref.k[:n].cpu().view(torch.int16))
    assert torch.equal(host.v[:n].view(torch.int16), ref.v[:n].cpu().view(torch.int16))


def test_host_copyback_with_cluster_summaries():
    """With clustered tail summaries the device output carries their metadata;
    the host copy holds the packed slots, counts and offsets, as documented."""
    K, V, Q = W.draw(WL, device="cuda")
    params = ck.certkv_default_params(tail_slot=0, tail_clusters=2)
    ref = ck.certkv_compress(K, V, Q, WL.B_live, params)
    hK, hV, hQ = K.cpu().pin_memory(), V.cpu().pin_memory(), Q.cpu().pin_memory()
    host = ck.Packed.empty_host(WL.B, WL.L, WL.H, WL.d, WL.B_live)
    got = ck.certkv_compress_host(hK, hV, hQ, WL.B_live, params, chunk=2, host_out=host)
    torch.cuda.synchronize()
    assert torch.equal(got.cluster_meta, ref.cluster_meta)
    assert torch.equal(host.offsets, ref.offsets.cpu())
    assert torch.equal(host.real_counts, ref.real_counts.cpu())
    n = int(ref.offsets[-1])
    assert torch.equal(host.positions[:n], ref.positions[:n].cpu())
    assert torch.equal(host.k[:n].view(torch.int16), ref.k[:n].cpu().view(torch.int16))
    assert torch.equal(host.v[:n].view(torch.int16), ref.v[:n].cpu().view(torch.int16))


@pytest.mark.parametrize("chunk", [1, 2, 0])
def test_host_pipeline_tiny_contexts(chunk):
    """The host-input pipeline on 5 (sequence, layer) pairs of 17-token
    contexts with 3 KV heads: chunks of one pair, of two (the last one short)
    and the automatic size all equal one device call bit for bit."""
    wl = W.Workload("T17", B=1, L=5, Hq=12, H=3, n=17, d=128, w=2, keep=(1, 3), kind="zipf")
    K, V, Q = W.draw(wl, device="cuda")
    params = ck.certkv_default_params()
    ref = _reference(K, V, Q, wl.B_live, params)
    got = ck.certkv_compress_host(K.cpu().pin_memory(), V.cpu().pin_memory(), Q.cpu().pin_memory(),
                                  wl.B_live, params, chunk=chunk, with_tail=True)
    torch.cuda.synchronize()
    _same(got, ref)
