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
    """One layer of a batch of sequences: packed cache + bf16 sink and window on the device.

    The sink and window live in one buffer of `sink + window + step + spare` rows per sequence
    as a contiguous block [sink | window] starting at row `y` (window tokens oldest first).  An
    append writes its new tokens in place after the window; a flush codes the oldest `step`
    window tokens (from their rows) and moves the block start up by the flushed count, copying
    only the sink rows; when the block would run past the buffer's end it is moved back to row 0
    once (every spare / step flushes).  The decode reads the block where it is, so no token is
    copied per append."""

    def __init__(self, plan, layer: int, batch: int, max_tokens: int, device, sink: int = 4,
                 window: int = 128, step: int = 16, spare_flushes: int = 64):
        import torch
        self.plan, self.layer, self.batch, self.max_tokens = plan, layer, batch, max_tokens
        self.state = SinkWindowState(sink, window, step)
        h = plan.dims.n_kv_heads
        self.cap = sink + window + step + step * max(0, spare_flushes)
        self.cache = plan.new_cache(batch, max_tokens, device)
        self.k_full = torch.zeros((batch, self.cap, h, HEAD_DIM), dtype=torch.bfloat16, device=device)
        self.v_full = torch.zeros_like(self.k_full)
        self.y = 0                      # first row of the [sink | window] block
        self.relocations = 0

    def _rows(self, a, b):
        return self.k_full[:, a:b], self.v_full[:, a:b]

    def append(self, k, v):
        """k, v: device bf16 [batch][m][H_kv][128], the next m tokens of every sequence."""
        import torch
        st = self.state
        S = st.sink
        m = k.shape[1]
        s0, n_win0 = st.n_sink, st.n_window
        to_sink, n_flush, pos = st.append(m)
        y = self.y
        if to_sink:
            self.k_full[:, y + s0:y + s0 + to_sink] = k[:, :to_sink]
            self.v_full[:, y + s0:y + s0 + to_sink] = v[:, :to_sink]
        r = m - to_sink
        kn, vn = k[:, to_sink:], v[:, to_sink:]
        if n_flush:
            # the oldest n_flush tokens of (old window ++ new tokens) go to the coded cache
            if pos + n_flush > self.max_tokens:
                raise ValueError("packed cache capacity exceeded")
            from_old = min(n_flush, n_win0)
            ko, vo = self._rows(y + S, y + S + from_old)
            if n_flush > from_old:
                kf = torch.cat([ko, kn[:, :n_flush - from_old]], dim=1)
                vf = torch.cat([vo, vn[:, :n_flush - from_old]], dim=1)
            else:
                kf, vf = ko.contiguous(), vo.contiguous()
            encode(self.plan, self.layer, kf, vf, self.cache, pos, self.max_tokens)
        if r == 0 and n_flush == 0:
            return
        old_keep = max(0, n_win0 - n_flush)          # old window tokens kept (the newest of them)
        new_keep = r - max(0, n_flush - n_win0)      # new tokens kept (the tail of the append)
        y1 = y + (n_win0 - old_keep)                 # the block start follows the kept tokens
        if y1 + S + old_keep + new_keep > self.cap:
            # move the block (sink and kept window tokens) back to row 0
            kb = torch.cat([self.k_full[:, y:y + S], self.k_full[:, y1 + S:y1 + S + old_keep]], dim=1)
            vb = torch.cat([self.v_full[:, y:y + S], self.v_full[:, y1 + S:y1 + S + old_keep]], dim=1)
            if S + old_keep + new_keep > self.cap:
                raise ValueError("append longer than the window buffer")
            self.k_full[:, :S + old_keep] = kb
            self.v_full[:, :S + old_keep] = vb
            y1 = 0
            self.relocations += 1
        elif y1 != y and S:
            ks, vs = self.k_full[:, y:y + S].clone(), self.v_full[:, y:y + S].clone()
            self.k_full[:, y1:y1 + S] = ks
            self.v_full[:, y1:y1 + S] = vs
        if new_keep:
            a = y1 + S + old_keep
            self.k_full[:, a:a + new_keep] = kn[:, r - new_keep:]
            self.v_full[:, a:a + new_keep] = vn[:, r - new_keep:]
        self.y = y1

    def decode(self, q, out=None, workspace=None, stream=None):
        st = self.state
        n_full = st.n_sink + st.n_window
        return decode_attention_sw(self.plan, self.layer, q, self.cache, st.sink, st.sink + st.n_coded,
                                   self.max_tokens, self.k_full, self.v_full, n_full, out=out, workspace=workspace,
                                   stream=stream, full_row0=self.y)
