"""Full-precision attention sink and recent window around the packed cache.

The paper's inference policy (Sec. 6 setup) keeps the first tokens of a sequence (4, the
attention sink) and a recent window (128 tokens, moved in steps of 16) in full precision and
transform-codes everything else.  Reading: the window fills up to window + step tokens; adding
the token that makes it window + step sends its oldest `step` tokens to the coded cache, so after
n tokens (n_sink, n_coded, n_window) follow the closed form of `SinkWindowState.counts`.

`SinkWindowState` is the host bookkeeping; `SinkWindowCache` keeps the bf16 sink and window of
one layer on the device, encodes flushed tokens with `encode` (at their absolute positions, so
the coded range is [sink, sink + n_coded)), and decodes with `decode_attention_sw`.
"""
from __future__ import annotations

from . import HEAD_DIM, decode_attention_sw, encode


class SinkWindowState:
    """Token accounting only: how many tokens are in the sink, coded, and in the window."""

    def __init__(self, sink: int = 4, window: int = 128, step: int = 16):
        if sink < 0 or window < 0 or step < 1:
            raise ValueError("sink, window >= 0 and step >= 1 required")
        self.sink, self.window, self.step = sink, window, step
        self.n_total = 0

    def counts(self, n: int):
        n_sink = min(n, self.sink)
        rest = n - n_sink
        n_coded = self.step * max(0, (rest - self.window) // self.step)
        return n_sink, n_coded, rest - n_coded

    @property
    def n_sink(self):
        return self.counts(self.n_total)[0]

    @property
    def n_coded(self):
        return self.counts(self.n_total)[1]

    @property
    def n_window(self):
        return self.counts(self.n_total)[2]

    def append(self, m: int):
        """Account for m new tokens.  Returns (to_sink, n_flush, coded_pos): the first `to_sink`
        new tokens go to the sink; then, of the old window followed by the remaining new tokens,
        the first `n_flush` (a multiple of step) are coded at positions [coded_pos, coded_pos +
        n_flush) and the rest is the new window."""
        s0, c0, _ = self.counts(self.n_total)
        self.n_total += m
        s1, c1, _ = self.counts(self.n_total)
        return s1 - s0, c1 - c0, self.sink + c0


class SinkWindowCache:
    """One layer of a batch of sequences: packed cache + bf16 sink and window on the device."""

    def __init__(self, plan, layer: int, batch: int, max_tokens: int, device, sink: int = 4,
                 window: int = 128, step: int = 16):
        import torch
        self.plan, self.layer, self.batch, self.max_tokens = plan, layer, batch, max_tokens
        self.state = SinkWindowState(sink, window, step)
        h = plan.dims.n_kv_heads
        cap = sink + window + step
        self.cache = plan.new_cache(batch, max_tokens, device)
        self.k_full = torch.zeros((batch, cap, h, HEAD_DIM), dtype=torch.bfloat16, device=device)
        self.v_full = torch.zeros_like(self.k_full)

    def append(self, k, v):
        """k, v: device bf16 [batch][m][H_kv][128], the next m tokens of every sequence."""
        import torch
        st = self.state
        s0, n_win0 = st.n_sink, st.n_window
        to_sink, n_flush, pos = st.append(k.shape[1])
        if to_sink:
            self.k_full[:, s0:s0 + to_sink] = k[:, :to_sink]
            self.v_full[:, s0:s0 + to_sink] = v[:, :to_sink]
        s = st.sink
        ks = torch.cat([self.k_full[:, s:s + n_win0], k[:, to_sink:]], dim=1)
        vs = torch.cat([self.v_full[:, s:s + n_win0], v[:, to_sink:]], dim=1)
        if n_flush:
            if pos + n_flush > self.max_tokens:
                raise ValueError("packed cache capacity exceeded")
            encode(self.plan, self.layer, ks[:, :n_flush].contiguous(), vs[:, :n_flush].contiguous(), self.cache,
                   pos, self.max_tokens)
        n_win = st.n_window
        self.k_full[:, s:s + n_win] = ks[:, n_flush:]
        self.v_full[:, s:s + n_win] = vs[:, n_flush:]

    def decode(self, q, out=None, workspace=None, stream=None):
        st = self.state
        n_full = st.n_sink + st.n_window
        return decode_attention_sw(self.plan, self.layer, q, self.cache, st.sink, st.sink + st.n_coded,
                                   self.max_tokens, self.k_full, self.v_full, n_full, out=out, workspace=workspace,
                                   stream=stream)
