"""The Python binding checks the device arguments whose sizes the C library cannot see (no GPU).

The required device type is pointed at the CPU so every check runs here; a call whose arguments
pass reaches the library with a null plan handle and is refused there, before any pointer is
read (its message names the C call alone), while a bad argument is refused by the binding (its
message says what was wrong)."""
import types

import pytest
import torch

bf16, f32 = torch.bfloat16, torch.float32
S = types.SimpleNamespace(cuda_stream=0)          # a stream handle without a CUDA context


@pytest.fixture
def fake(aatc, monkeypatch):
    monkeypatch.setattr(aatc, "_DEVICE_TYPE", "cpu")
    dm = aatc.dims(2, 2, 8)
    plan = types.SimpleNamespace(dims=dm, handle=None, cache_bytes=lambda b, m: 4 * 1000 * b * m,
                                 workspace_bytes=lambda b, n: 1024)
    return aatc, plan


def _library_refused(e, call):
    assert e.value.status == 1 and str(e.value).startswith(f"{call}: "), str(e.value)


def _binding_refused(e, call, what):
    assert e.value.status == 1 and str(e.value).startswith(f"{call} (") and what in str(e.value), str(e.value)


def test_encode(fake):
    aatc, plan = fake
    K = torch.zeros((1, 5, 2, 128), dtype=bf16)
    cache = torch.zeros(1000 * 64, dtype=torch.int32)
    with pytest.raises(aatc.AatcError) as e:
        aatc.encode(plan, 0, K, K.clone(), cache, 0, 64, stream=S)
    _library_refused(e, "aatc_encode")
    with pytest.raises(aatc.AatcError) as e:                       # empty append: still a valid shape
        aatc.encode(plan, 0, K[:, :0], K[:, :0], cache, 0, 64, stream=S)
    _library_refused(e, "aatc_encode")
    for bad_k, bad_v, what in ((K.float(), K, "K must be torch.bfloat16"),
                               (torch.zeros((1, 5, 3, 128), dtype=bf16), K, "K size 2 must be 2"),
                               (torch.zeros((5, 2, 128), dtype=bf16), K, "K must have 4 dimensions"),
                               (K, torch.zeros((1, 4, 2, 128), dtype=bf16), "V size 1 must be 5")):
        with pytest.raises(aatc.AatcError) as e:
            aatc.encode(plan, 0, bad_k, bad_v, cache, 0, 64, stream=S)
        _binding_refused(e, "aatc_encode", what)
    with pytest.raises(aatc.AatcError) as e:                       # cache smaller than (1, 65) needs
        aatc.encode(plan, 0, K, K, cache, 0, 65, stream=S)
    _binding_refused(e, "aatc_encode", "needed)")


def test_encode_hidden(fake):
    aatc, plan = fake
    x = torch.zeros((1, 7, 256), dtype=bf16)
    a_hat = torch.zeros((2, 2, 2, 128, 256), dtype=bf16)
    cache = torch.zeros(1000 * 64, dtype=torch.int32)
    with pytest.raises(aatc.AatcError) as e:
        aatc.encode_hidden(plan, 0, x, a_hat, cache, 0, 64, stream=S)
    _library_refused(e, "aatc_encode_hidden")
    with pytest.raises(aatc.AatcError) as e:
        aatc.encode_hidden(plan, 0, x[:, :, :128].contiguous(), a_hat, cache, 0, 64, stream=S)
    _binding_refused(e, "aatc_encode_hidden", "a_hat must be")


def test_decode_and_prefill(fake):
    aatc, plan = fake
    cache = torch.zeros(1000 * 2 * 64, dtype=torch.int32)
    q = torch.zeros((2, 8, 128), dtype=bf16)
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention(plan, 0, q, cache, 64, 64, workspace=torch.zeros(256), stream=S)
    _library_refused(e, "aatc_decode_attention")
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention_noalloc(plan, 0, q, torch.zeros((2, 8, 128)), cache, 64, 64, stream=S)
    _library_refused(e, "aatc_decode_attention_noalloc")
    for bad, what in ((q.float(), "q must be torch.bfloat16"), (q[:, :4].contiguous(), "q size 1 must be 8")):
        with pytest.raises(aatc.AatcError) as e:
            aatc.decode_attention(plan, 0, bad, cache, 64, 64, stream=S)
        _binding_refused(e, "aatc_decode_attention", what)
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention(plan, 0, q, cache, 64, 64, out=torch.zeros((2, 8, 127)), stream=S)
    _binding_refused(e, "aatc_decode_attention", "values")
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention(plan, 0, q, cache, 64, 64, out=torch.zeros((2, 8, 128), dtype=torch.float64), stream=S)
    _binding_refused(e, "aatc_decode_attention", "out must be a cpu tensor of torch.float32")
    qp = torch.zeros((2, 3, 8, 128), dtype=bf16)
    with pytest.raises(aatc.AatcError) as e:
        aatc.prefill_attention(plan, 0, qp, 0, cache, 64, 64, stream=S)
    _library_refused(e, "aatc_prefill_workspace_bytes")
    with pytest.raises(aatc.AatcError) as e:
        aatc.prefill_attention(plan, 0, qp[:, :, :4].contiguous(), 0, cache, 64, 64, stream=S)
    _binding_refused(e, "aatc_prefill_attention", "q size 2 must be 8")


def test_sink_window_and_dequantize(fake):
    aatc, plan = fake
    cache = torch.zeros(1000 * 64, dtype=torch.int32)
    q = torch.zeros((1, 8, 128), dtype=bf16)
    kf = torch.zeros((1, 20, 2, 128), dtype=bf16)
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention_sw(plan, 0, q, cache, 4, 40, 64, kf, kf.clone(), 20, stream=S)
    _library_refused(e, "aatc_decode_attention_sw")
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention_sw(plan, 0, q, cache, 4, 40, 64, kf, None, 20, stream=S)
    _binding_refused(e, "aatc_decode_attention_sw", "v_full must be")
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention_sw(plan, 0, q, cache, 4, 40, 64, kf[:, :, :1].contiguous(), kf[:, :, :1].contiguous(), 2, stream=S)
    _binding_refused(e, "aatc_decode_attention_sw", "k_full size 2 must be 2")
    with pytest.raises(aatc.AatcError) as e:
        aatc.dequantize(plan, 0, cache, 1, 0, 10, 64, stream=S)
    _library_refused(e, "aatc_dequantize")
    with pytest.raises(aatc.AatcError) as e:
        aatc.dequantize(plan, 0, cache, 2, 0, 10, 64, stream=S)
    _binding_refused(e, "aatc_dequantize", "needed)")


def test_bf16_reference_decode(fake):
    aatc, _ = fake
    K = torch.zeros((2, 50, 2, 128), dtype=bf16)
    q = torch.zeros((2, 8, 128), dtype=bf16)
    with pytest.raises(aatc.AatcError) as e:                       # the C call refuses n_ctx > max_tokens
        aatc.bf16_decode_attention(K, K.clone(), q, 51, workspace=torch.zeros(1 << 16), stream=S)
    assert str(e.value).startswith("aatc_bf16_decode_attention: ")
    with pytest.raises(aatc.AatcError) as e:
        aatc.bf16_decode_attention(K, K.clone(), q[:1].contiguous(), 50, workspace=torch.zeros(1 << 16), stream=S)
    _binding_refused(e, "aatc_bf16_decode_attention", "q size 0 must be 2")
