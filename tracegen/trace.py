"""Seeded synthetic request traces (input generation only).

A trace is per-request metadata built on the host with numpy:
  * prompt length L[r] (uint32 tokens) and arrival time arrival_us[r];
  * the prompt's token content, described as a list of *pieces*
    (stream id, start position, length): the prompt is the concatenation of
    its pieces, and a piece's tokens are drawn from a counter-based generator
        token(stream, pos) = mix64(token_seed ^ stream*PHI ^ pos) mod vocab,
    mix64 being one SplitMix64 output step (Steele, Lea & Flood, OOPSLA 2014).
    Requests that share a prefix share the piece (same stream, same positions)
    and hence the same tokens;
  * consecutive batches of `batch` requests, and (scaling workload) the
    add/remove events applied between batches.

Random draws (lengths, Zipf ranks, arrivals, the id an event removes) come
from numpy's PCG64 seeded with the workload seed.  Token content is a pure
function of (token_seed, stream, pos), so host (numpy, here) and device
(gen_tokens.cu) produce identical tokens without transferring them.

Nothing here computes any part of the routing method.
"""

import numpy as np

PHI = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)

# Stream-id namespaces: shared prefixes, per-request unique parts, session chunks.
STREAM_PREFIX = 1
STREAM_UNIQUE = 1 << 40
STREAM_SESSION = 1 << 41

ALIGN_TOKENS = 4  # prompts start on 16-byte boundaries in a batch buffer


def mix64(x):
    """One SplitMix64 output step applied to state x (uint64 numpy array)."""
    with np.errstate(over="ignore"):
        z = x + PHI
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        return z ^ (z >> np.uint64(31))


def piece_tokens(token_seed, vocab, stream, start, length):
    """Tokens of one piece as a uint32 array."""
    pos = np.arange(start, start + length, dtype=np.uint64)
    with np.errstate(over="ignore"):
        x = np.uint64(token_seed) ^ (np.uint64(stream) * PHI) ^ pos
    return (mix64(x) % np.uint64(vocab)).astype(np.uint32)


def _zipf_sampler(n, s, rng, size):
    """Ranks 0..n-1 with P(k) proportional to (k+1)^-s (inverse-CDF table)."""
    w = np.arange(1, n + 1, dtype=np.float64) ** (-float(s))
    cdf = np.cumsum(w)
    cdf /= cdf[-1]
    u = rng.random(size)
    return np.minimum(np.searchsorted(cdf, u, side="right"), n - 1).astype(np.int64)


def round_up(x, a):
    return (x + a - 1) // a * a


class Trace:
    """Per-request metadata of one synthetic workload."""

    def __init__(self, cfg, n_requests=None, seed=None):
        self.cfg = dict(cfg)
        if n_requests is not None:
            self.cfg["n_requests"] = int(n_requests)
        if seed is not None:
            self.cfg["seed"] = int(seed)
        c = self.cfg
        self.seed = int(c["seed"])
        self.token_seed = int(mix64(np.array([self.seed ^ 0x70CE], dtype=np.uint64))[0])
        self.vocab = int(c["vocab"])
        rng = np.random.Generator(np.random.PCG64(self.seed))
        n = int(c["n_requests"])
        builder = {
            "prefix_suffix": self._gen_prefix_suffix,
            "template": self._gen_template,
            "fixed_prefix": self._gen_fixed_prefix,
            "sessions": self._gen_sessions,
        }[c["kind"]]
        pr, ps, pst, pl, uncached = builder(rng, n)
        self.piece_req = np.asarray(pr, dtype=np.int64)
        self.piece_stream = np.asarray(ps, dtype=np.uint64)
        self.piece_start = np.asarray(pst, dtype=np.uint64)
        self.piece_len = np.asarray(pl, dtype=np.int64)
        order = np.argsort(self.piece_req, kind="stable")
        for a in ("piece_req", "piece_stream", "piece_start", "piece_len"):
            setattr(self, a, getattr(self, a)[order])
        self.n = n
        self.L = np.bincount(self.piece_req, weights=self.piece_len, minlength=n).astype(np.int64)
        self.req_piece_off = np.zeros(n + 1, dtype=np.int64)
        np.cumsum(np.bincount(self.piece_req, minlength=n), out=self.req_piece_off[1:])
        # Poisson arrivals at load rho: mean gap = cost * E[uncached] / (rho * N) us.
        mean_gap = c["cost_us"] * float(np.mean(uncached)) / (c["rho"] * c["n_instances"])
        u = rng.random(n)
        gaps = np.floor(-np.log1p(-u) * mean_gap).astype(np.int64)
        self.arrival_us = np.cumsum(gaps).astype(np.uint64)
        self.batch = int(c["batch"])
        self.batches = [(s, min(s + self.batch, n)) for s in range(0, n, self.batch)]
        self.events = self._gen_events(rng)
        # Global layout of all prompts in one buffer, each start 16-byte aligned.
        self.req_off = np.zeros(n + 1, dtype=np.int64)
        np.cumsum(round_up(self.L, ALIGN_TOKENS), out=self.req_off[1:])

    # -- prompt structures -------------------------------------------------
    def _gen_prefix_suffix(self, rng, n):
        c = self.cfg
        plen = rng.integers(c["prefix_lo"], c["prefix_hi"], size=c["n_prefix"], endpoint=True)
        L = rng.integers(c["len_lo"], c["len_hi"], size=n, endpoint=True)
        p = _zipf_sampler(c["n_prefix"], c["zipf_s"], rng, n)
        shared = np.minimum(plen[p], L)
        rest = L - shared
        r = np.arange(n)
        pr = np.concatenate([r, r[rest > 0]])
        ps = np.concatenate([STREAM_PREFIX + p, STREAM_UNIQUE + r[rest > 0]])
        pst = np.zeros(len(pr), dtype=np.int64)
        pl = np.concatenate([shared, rest[rest > 0]])
        return pr, ps, pst, pl, rest

    def _gen_template(self, rng, n):
        c = self.cfg
        plen = rng.integers(c["prefix_lo"], c["prefix_hi"], size=c["n_prefix"], endpoint=True)
        p = _zipf_sampler(c["n_prefix"], c["zipf_s"], rng, n)
        u = rng.integers(c["uniq_lo"], c["uniq_hi"], size=n, endpoint=True)
        r = np.arange(n)
        pr = np.concatenate([r, r])
        ps = np.concatenate([STREAM_PREFIX + p, STREAM_UNIQUE + r])
        pst = np.zeros(2 * n, dtype=np.int64)
        pl = np.concatenate([plen[p], u])
        return pr, ps, pst, pl, u

    def _gen_fixed_prefix(self, rng, n):
        c = self.cfg
        L = rng.integers(c["len_lo"], c["len_hi"], size=n, endpoint=True)
        p = _zipf_sampler(c["n_prefix"], c["zipf_s"], rng, n)
        shared = np.minimum(c["prefix_len"], L)
        rest = L - shared
        r = np.arange(n)
        pr = np.concatenate([r, r[rest > 0]])
        ps = np.concatenate([STREAM_PREFIX + p, STREAM_UNIQUE + r[rest > 0]])
        pst = np.zeros(len(pr), dtype=np.int64)
        pl = np.concatenate([shared, rest[rest > 0]])
        return pr, ps, pst, pl, rest

    def _gen_sessions(self, rng, n):
        """Concurrent sessions; turn t's prompt = all earlier chunks + chunk t.

        A finished session (its drawn turn count reached, or its next prompt
        would pass max_prompt) is replaced by a fresh one until n requests
        have been emitted.  The next session to speak is uniform among the
        active ones."""
        c = self.cfg
        S = int(c["n_sessions"])
        turns = np.minimum(rng.geometric(c["turn_p"], size=S), c["max_turns"])
        sess_id = np.arange(S, dtype=np.int64)
        next_id = S
        done = np.zeros(S, dtype=np.int64)
        hist = [[] for _ in range(S)]       # list of chunk lengths per slot
        hist_len = np.zeros(S, dtype=np.int64)
        pr, ps, pl, chunks = [], [], [], []
        r = 0
        picks = rng.integers(0, S, size=4 * n + 16)
        chunk_draw = rng.integers(c["chunk_lo"], c["chunk_hi"], size=4 * n + 16, endpoint=True)
        k = 0
        while r < n:
            if k >= len(picks):
                picks = rng.integers(0, S, size=4 * n + 16)
                chunk_draw = rng.integers(c["chunk_lo"], c["chunk_hi"], size=4 * n + 16, endpoint=True)
                k = 0
            s = int(picks[k]); ch = int(chunk_draw[k]); k += 1
            if done[s] >= turns[s] or hist_len[s] + ch > c["max_prompt"]:
                sess_id[s] = next_id; next_id += 1
                turns[s] = min(int(rng.geometric(c["turn_p"])), c["max_turns"])
                done[s] = 0; hist[s] = []; hist_len[s] = 0
                continue
            hist[s].append(ch)
            base = STREAM_SESSION + int(sess_id[s]) * 64
            for t, ln in enumerate(hist[s]):
                pr.append(r); ps.append(base + t); pl.append(ln)
            hist_len[s] += ch
            done[s] += 1
            chunks.append(ch)
            r += 1
        pst = np.zeros(len(pr), dtype=np.int64)
        return pr, ps, pst, pl, np.asarray(chunks)

    def _gen_events(self, rng):
        """(batch index, 'add'|'remove', id): every scale_every requests,
        alternately add the next fresh id and remove a uniformly chosen live id,
        applied before the first batch starting at or after the threshold."""
        c = self.cfg
        every = int(c.get("scale_every", 0))
        if every <= 0:
            return []
        live = list(range(c["n_instances"]))
        fresh = c["n_instances"]
        ev = []
        k = 1
        while k * every < self.n:
            thr = k * every
            b = next(i for i, (s, _) in enumerate(self.batches) if s >= thr)
            if k % 2 == 1:
                ev.append((b, "add", fresh)); live.append(fresh); fresh += 1
            else:
                victim = live[int(rng.integers(0, len(live)))]
                ev.append((b, "remove", victim)); live.remove(victim)
            k += 1
        return ev

    # -- token content -------------------------------------------------------
    def max_instance_id(self):
        ids = [e[2] for e in self.events if e[1] == "add"]
        return max([self.cfg["n_instances"] - 1] + ids)

    def request_tokens(self, r):
        out = []
        for i in range(self.req_piece_off[r], self.req_piece_off[r + 1]):
            out.append(piece_tokens(self.token_seed, self.vocab, int(self.piece_stream[i]),
                                    int(self.piece_start[i]), int(self.piece_len[i])))
        return np.concatenate(out) if out else np.zeros(0, np.uint32)

    def batch_layout(self, b):
        """(start, end, offsets[n] relative to the batch, lengths[n], n_tokens)."""
        s, e = self.batches[b]
        off = (self.req_off[s:e] - self.req_off[s]).astype(np.uint64)
        return s, e, off, self.L[s:e].astype(np.uint32), int(self.req_off[e] - self.req_off[s])

    def batch_tokens(self, b):
        """Host token buffer of batch b in the aligned batch layout."""
        s, e, off, lens, ntok = self.batch_layout(b)
        buf = np.zeros(ntok, dtype=np.uint32)
        for i, r in enumerate(range(s, e)):
            buf[int(off[i]):int(off[i]) + int(lens[i])] = self.request_tokens(r)
        return buf

    def batch_time(self, b):
        """Batch time: the arrival of the batch's last request."""
        return int(self.arrival_us[self.batches[b][1] - 1])

    def pieces_for_range(self, r0, r1):
        """Piece descriptors (dst token offset relative to req r0's start,
        stream, start, length) of requests [r0, r1), for the device filler."""
        p0, p1 = self.req_piece_off[r0], self.req_piece_off[r1]
        req = self.piece_req[p0:p1]
        within = np.zeros(p1 - p0, dtype=np.int64)
        if p1 > p0:
            lens = self.piece_len[p0:p1]
            cum = np.cumsum(lens) - lens
            first = self.req_piece_off[req] - p0
            within = cum - cum[first]
        dst = (self.req_off[req] - self.req_off[r0]) + within
        return (dst.astype(np.uint64), self.piece_stream[p0:p1].copy(),
                self.piece_start[p0:p1].astype(np.uint64), self.piece_len[p0:p1].astype(np.uint32))
