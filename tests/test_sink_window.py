"""Full-precision attention sink and recent window (NEXT row 1; Sec. 6 setup: 4 sink tokens, a
128-token window moved in steps of 16): the oracle's joint softmax pinned against plain
attention, the token accounting against a step-by-step simulation, and the cache manager's
bookkeeping on the host."""
import math

import numpy as np
import pytest

from oracle import aatc_oracle as O


def _orthonormal(rng, d=128):
    q, r = np.linalg.qr(rng.standard_normal((d, d)))
    return q * np.sign(np.diag(r))


def test_mixed_decode_is_plain_attention_when_coding_is_lossless():
    """With exact coefficients h = U^T k (no quantization), splitting the tokens into a coded part
    and an uncompressed part, in any proportion, gives plain single-query attention over all of
    them (orthonormal U: q.k = (U^T q).(U^T k), and the value transform is linear)."""
    rng = np.random.default_rng(11)
    H, G, n = 2, 3, 300
    uk = np.stack([_orthonormal(rng) for _ in range(H)])
    uv = np.stack([_orthonormal(rng) for _ in range(H)])
    k = rng.standard_normal((H, n, 128)) * 2.0
    v = rng.standard_normal((H, n, 128))
    q = rng.standard_normal((H * G, 128))
    want = np.stack([O.attention(q[j], k[j // G], v[j // G]) for j in range(H * G)])
    for n_coded in (0, 1, 137, 296, 300):
        hk = np.einsum("hnd,hdc->hnc", k[:, :n_coded], uk)
        hv = np.einsum("hnd,hdc->hnc", v[:, :n_coded], uv)
        got = O.decode_attention_mixed(q, hk, hv, uk, uv, G, k[:, n_coded:], v[:, n_coded:])
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


def test_mixed_decode_without_full_tokens_is_the_coded_decode():
    rng = np.random.default_rng(12)
    H, G, n = 1, 4, 50
    uk, uv = _orthonormal(rng)[None], _orthonormal(rng)[None]
    hk, hv = rng.standard_normal((H, n, 128)), rng.standard_normal((H, n, 128))
    q = rng.standard_normal((G, 128))
    empty = np.zeros((H, 0, 128))
    np.testing.assert_allclose(O.decode_attention_mixed(q, hk, hv, uk, uv, G, empty, empty),
                               O.decode_attention(q, hk, hv, uk, uv, G), rtol=1e-13, atol=1e-13)


def _simulate(n_tokens, sink=4, window=128, step=16):
    n_sink = n_coded = n_win = 0
    for _ in range(n_tokens):
        if n_sink < sink:
            n_sink += 1
            continue
        n_win += 1
        if n_win == window + step:
            n_win -= step
            n_coded += step
    return n_sink, n_coded, n_win


@pytest.mark.parametrize("sink,window,step", [(4, 128, 16), (0, 32, 8), (2, 16, 16)])
def test_sink_window_counts_match_token_by_token_policy(sink, window, step):
    for n in range(0, 700):
        assert O.sink_window_counts(n, sink, window, step) == _simulate(n, sink, window, step), n


def test_cache_manager_bookkeeping_matches_policy():
    """The package's host bookkeeping applies the same schedule: each append codes a multiple of
    the step, oldest window tokens first, at the next coded positions."""
    from paper_2608_14191_gb300.sink_window import SinkWindowState
    st = SinkWindowState(sink=4, window=128, step=16)
    n, pos = 0, 4
    for m in (1, 3, 7, 200, 16, 15, 1, 1, 40, 333, 0, 5000):
        to_sink, n_flush, at = st.append(m)
        n += m
        assert (st.n_sink, st.n_coded, st.n_window) == O.sink_window_counts(n)
        assert n_flush % 16 == 0 and at == pos
        assert to_sink == O.sink_window_counts(n)[0] - O.sink_window_counts(n - m)[0]
        pos += n_flush
    assert pos == 4 + st.n_coded


class _FakePlan:
    """Just enough of a Plan for the cache manager's host logic on CPU tensors."""

    class dims:
        n_kv_heads = 2

    def new_cache(self, batch, max_tokens, device):
        import torch
        return torch.zeros(8, dtype=torch.int32)


@pytest.mark.parametrize("spare", [64, 1])
def test_cache_manager_keeps_sink_and_window_in_place(monkeypatch, spare):
    """SinkWindowCache on CPU tensors with the encode call recorded: after every append the block
    [y, y + n_sink + n_window) holds the sink tokens and then the newest window tokens in order,
    the flushed tokens are exactly the coded positions in order, and appends of one token copy
    no window token (only a flush moves the four sink rows, and the block is moved back to row 0
    once every `spare` flushes)."""
    import torch
    import paper_2608_14191_gb300.sink_window as sw
    coded = []

    def fake_encode(plan, layer, k, v, cache, pos, max_tokens):
        assert k.is_contiguous() and v.is_contiguous() and torch.equal(k, v - 0.5)
        assert pos == 4 + sum(c.shape[1] for c in coded)
        coded.append(k.clone())

    monkeypatch.setattr(sw, "encode", fake_encode)
    batch, H, n_max = 2, 2, 3000
    tok = torch.arange(batch * n_max, dtype=torch.float32).reshape(batch, n_max, 1, 1).expand(batch, n_max, H, 128)
    swc = sw.SinkWindowCache(_FakePlan(), 0, batch, n_max, "cpu", spare_flushes=spare)
    swc.k_full = swc.k_full.float()
    swc.v_full = swc.v_full.float()
    n = 0
    for m in [1, 2, 1, 200, 16, 15, 1, 1, 40, 333] + [1] * 300 + [17, 5, 900]:
        swc.append(tok[:, n:n + m].contiguous(), tok[:, n:n + m].contiguous() + 0.5)
        n += m
        st = swc.state
        assert (st.n_sink, st.n_coded, st.n_window) == O.sink_window_counts(n)
        want = list(range(st.n_sink)) + list(range(st.sink + st.n_coded, n))
        blk = swc.k_full[:, swc.y:swc.y + len(want), 0, 0]
        assert torch.equal(blk, tok[:, want, 0, 0]), n
        assert torch.equal(swc.v_full[:, swc.y:swc.y + len(want), 0, 0], blk + 0.5)
    got = torch.cat(coded, dim=1)[:, :, 0, 0]
    assert torch.equal(got, tok[:, 4:4 + swc.state.n_coded, 0, 0])
    if spare == 64:
        assert swc.relocations <= 1 + swc.state.n_coded // (16 * 64)
