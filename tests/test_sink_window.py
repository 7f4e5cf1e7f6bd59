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
