"""GPU parity of the encode from hidden states (Sec. 5 Step 1: the cache holds the coefficients of
x A) against the oracle, through the C ABI: codes, token scales and decode attention over the
cache it writes."""
import numpy as np
import pytest
import torch

import harness as Hn
from oracle import aatc_oracle as O
import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
SEED = 1002


class HiddenCase:
    """A layer whose keys / values are projections x W of hidden states: the plan is calibrated on
    the calibration keys / values K = X W, and the encode operand is W U in bf16."""

    def __init__(self, aatc, d_model, n_kv, n_q, avg_bits=2.75, n_calib=4096):
        self.d_model, self.n_kv, self.n_q = d_model, n_kv, n_q
        self.cfg = W.Config(9, f"hidden_{d_model}", 1, n_kv, n_q, 1, 0, (avg_bits,), 1, "hidden-state encode")
        x_cal = W.hidden_states(SEED, 0, d_model, n_calib).astype(np.float64)
        self.w_k = W.projection_weight(SEED, 0, 0, d_model, n_kv)
        self.w_v = W.projection_weight(SEED, 0, 1, d_model, n_kv)
        ck = np.stack([(x_cal @ self.w_k[:, h * 128:(h + 1) * 128]) for h in range(n_kv)])[None]
        cv = np.stack([(x_cal @ self.w_v[:, h * 128:(h + 1) * 128]) for h in range(n_kv)])[None]
        cq = np.stack([W.calibration_queries(self.cfg, 0, j) for j in range(n_q)])[None]
        self.dm = aatc.dims(1, n_kv, n_q)
        p = aatc.calibrate(self.dm, ck.astype(np.float32), cv.astype(np.float32), cq, avg_bits)
        self.basis, self.bits, self.scales = p["basis"], p["bits"], p["scales"]
        self.plan = aatc.Plan(self.dm, self.basis, self.bits, self.scales)
        self.basis_bf16 = Hn.bf16_round(self.basis)
        ah = aatc.hidden_operand(self.dm, self.w_k[None], self.w_v[None], self.basis)
        self.a_hat_host = torch.from_numpy(ah.view(np.int16)).view(torch.bfloat16).float().numpy()
        self.a_hat = torch.from_numpy(ah.view(np.int16)).view(torch.bfloat16).to(DEV).contiguous()

    def stream(self, layer, head, kind):
        return self.basis[layer, head, kind], self.bits[layer, head, kind], self.scales[layer, head, kind]


def _check_all(case, cache, x_host, batch, max_tokens, t0, n):
    u32 = cache.cpu().numpy().view(np.uint32)
    stats = {"codes": 0, "mismatch": 0}
    for b in range(batch):
        for h in range(case.n_kv):
            for kind in (0, 1):
                rec, alpha = O.cache_records(u32, batch, case.n_kv, max_tokens, case.plan.n_words, b, h, kind, t0, n)
                s = Hn.check_codes(case, 0, h, kind, x_host[b], rec, alpha,
                                   encode_matrix=case.a_hat_host[0, h, kind].T)
                stats["codes"] += s["codes"]
                stats["mismatch"] += s["mismatch"]
                Hn.NearThreshold.add("hidden-state encode (small cases)", s["mismatch"], s["codes"], s["near"])
    Hn.NearThreshold.assert_bound("hidden-state encode (small cases)")
    return u32


@pytest.mark.parametrize("d_model", [256, 640])
def test_encode_hidden_codes(aatc, d_model):
    case = HiddenCase(aatc, d_model, n_kv=2, n_q=8)
    batch, n_tok, max_tokens = 2, 300, 384                  # two full tiles and a ragged one
    x = W.hidden_states_device(SEED, 0, d_model, batch, n_tok, DEV)
    cache = case.plan.new_cache(batch, max_tokens, DEV)
    cache.zero_()
    aatc.encode_hidden(case.plan, 0, x, case.a_hat, cache, 0, max_tokens)
    torch.cuda.synchronize()
    _check_all(case, cache, x.float().cpu().numpy(), batch, max_tokens, 0, n_tok)
    assert case.plan.device_error() == 0


def test_encode_hidden_append_at_odd_position_and_decode(aatc):
    """Appends at a position that is not a tile or quad boundary leave earlier tokens intact, and
    decode attention over the resulting cache matches the oracle's attention over the GPU's codes."""
    d_model = 384
    case = HiddenCase(aatc, d_model, n_kv=2, n_q=8)
    batch, max_tokens = 1, 512
    x = W.hidden_states_device(SEED, 0, d_model, batch, 450, DEV)
    cache = case.plan.new_cache(batch, max_tokens, DEV)
    cache.zero_()
    aatc.encode_hidden(case.plan, 0, x[:, :133].contiguous(), case.a_hat, cache, 0, max_tokens)
    aatc.encode_hidden(case.plan, 0, x[:, 133:].contiguous(), case.a_hat, cache, 133, max_tokens)
    torch.cuda.synchronize()
    u32 = _check_all(case, cache, x.float().cpu().numpy(), batch, max_tokens, 0, 450)
    qs = W.queries_host(case.cfg, 0, batch, 1)
    q = torch.from_numpy(qs[0]).to(DEV).to(torch.bfloat16)
    out = aatc.decode_attention(case.plan, 0, q, cache, 450, max_tokens).cpu().numpy()
    ref = Hn.oracle_decode_from_cache(case, u32, batch, max_tokens, 0, 0, qs[0, 0], 450)
    Hn.check_decode(out[0], np.stack([ref[j] for j in range(case.n_q)]))


def test_encode_hidden_argument_errors(aatc):
    case = HiddenCase(aatc, 128, n_kv=1, n_q=4, n_calib=2048)
    x = torch.zeros((1, 10, 128), dtype=torch.bfloat16, device=DEV)
    cache = case.plan.new_cache(1, 64, DEV)
    with pytest.raises(aatc.AatcError):
        aatc.encode_hidden(case.plan, 0, x[:, :, :96].contiguous(), case.a_hat, cache, 0, 64)   # d_model % 64
    with pytest.raises(aatc.AatcError):
        aatc.encode_hidden(case.plan, 0, x, case.a_hat, cache, 60, 64)                        # capacity
    with pytest.raises(aatc.AatcError):
        aatc.encode_hidden(case.plan, 1, x, case.a_hat, cache, 0, 64)                         # layer


def test_encode_hidden_llama_shape_sampled(aatc):
    """Bench configuration: Llama-3.1-8B-shaped layer input (d_model 4096, 8 kv-heads), 32768
    tokens in the launch the bench times; codes and scales of every kv-head compared on 256
    sampled tokens (the oracle's fp64 projection over d_model 4096 is the slow part)."""
    d_model, n_kv, n_tok = 4096, 8, 32768
    case = HiddenCase(aatc, d_model, n_kv=n_kv, n_q=32)
    x = W.hidden_states_device(SEED, 0, d_model, 1, n_tok, DEV)
    cache = case.plan.new_cache(1, n_tok, DEV)
    aatc.encode_hidden(case.plan, 0, x, case.a_hat, cache, 0, n_tok)
    torch.cuda.synchronize()
    assert case.plan.device_error() == 0
    u32 = cache.cpu().numpy().view(np.uint32)
    rng = np.random.default_rng(7)
    toks = np.sort(rng.choice(n_tok, 256, replace=False))
    xs = x[0, torch.from_numpy(toks).to(DEV)].float().cpu().numpy()
    total = mis = 0
    for h in range(n_kv):
        for kind in (0, 1):
            rec_all, alpha_all = O.cache_records(u32, 1, n_kv, n_tok, case.plan.n_words, 0, h, kind, 0, n_tok)
            s = Hn.check_codes(case, 0, h, kind, xs, rec_all[toks], alpha_all[toks],
                               encode_matrix=case.a_hat_host[0, h, kind].T)
            total += s["codes"]
            mis += s["mismatch"]
            Hn.NearThreshold.add("hidden-state encode (Llama layer input, 256 tokens x 8 kv-heads)", s["mismatch"],
                                 s["codes"], s["near"])
    Hn.NearThreshold.assert_bound("hidden-state encode (Llama layer input, 256 tokens x 8 kv-heads)")
