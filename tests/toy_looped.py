"""A toy looped Transformer for end-to-end checks of verification, greedy
acceptance and the commit (Sec. 3.4, App. B.1, the greedy target-preservation
proposition of App. B).  Test infrastructure only.

The model: token embedding E, L core layers applied R times (recurrent
depths 1..R); at depth r layer l the position's hidden state h gives q, k, v
(rounded to bf16, the cache's storage type), attention reads the verified
prefix's K/V at depth r (the target's own depth, kappa = nu = r) plus the
block's own K/V under the causal mask, and h <- h + tanh(o Wo).  The readout
is logits = h(R) U.  Random weights from a seed; with these scales the
greedy continuation is varied and depends on every context token (changing
one prompt token changes the whole continuation).

Two implementations of the same model:
  ToyLoopedCPU  fp64 numpy, attention by the oracle (test infrastructure);
  ToyLoopedGPU  fp64 torch on the GPU for the projections (so q, k, v round
                to the same bf16 values as on the CPU while the hidden
                states agree), attention, acceptance and the commit through
                the library (das_verify_attention, das_greedy_accept,
                das_kv_append).
Both decode autoregressively (ar) or speculatively (spec: a block [anchor,
y_1 .. y_{w-1}] verified in one pass, the longest agreeing prefix accepted,
n = min(a + 1, w) inputs committed)."""
import numpy as np


def to_bf16_bits(x):
    """float -> bf16 bits, round to nearest even (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def bf16_bits_to_f64(b):
    return (np.asarray(b, dtype=np.uint32) << 16).view(np.float32).astype(np.float64)


class Weights:
    """qk / v: scales of the query-key and value projections (relative to
    1/sqrt(d)); larger qk sharpens attention and makes the continuation more
    sensitive to small changes of the attention outputs."""

    def __init__(self, seed, V=64, d=32, H=2, D=64, L=2, R=4, qk=2.0, v=1.0):
        rng = np.random.default_rng(seed)
        self.V, self.d, self.H, self.D, self.L, self.R = V, d, H, D, L, R
        self.E = rng.normal(0, 1, (V, d))
        s = 1.0 / np.sqrt(d)
        self.Wq = rng.normal(0, qk * s, (L, d, H * D))
        self.Wk = rng.normal(0, qk * s, (L, d, H * D))
        self.Wv = rng.normal(0, v * s, (L, d, H * D))
        self.Wo = rng.normal(0, 1.0 / np.sqrt(H * D), (L, H * D, d))
        self.U = np.random.default_rng(seed + 100).normal(0, 1, (d, V))


class ToyLoopedCPU:
    """bf16_outputs: round every attention output to bf16 (the library's
    output type) before the residual update, to measure how much that
    rounding alone moves the logits."""

    def __init__(self, w, cap, bf16_outputs=False):
        import oracle
        self.o, self.w, self.cap = oracle, w, cap
        self.bf16_outputs = bf16_outputs
        shape = (w.R, w.L, 1, cap, w.H, w.D)
        self.K = np.zeros(shape, np.uint16)
        self.V = np.zeros(shape, np.uint16)
        self.P = 0

    def forward(self, tokens):
        """Block forward at positions P .. P+T-1: (logits fp32 [T][V], staged K, V)."""
        w, T = self.w, len(tokens)
        h = w.E[np.asarray(tokens)]
        sk = np.zeros((w.R, w.L, 1, T, w.H, w.D), np.uint16)
        sv = np.zeros_like(sk)
        for r in range(1, w.R + 1):
            for l in range(w.L):
                q = to_bf16_bits(h @ w.Wq[l]).reshape(1, T, w.H, w.D)
                k = to_bf16_bits(h @ w.Wk[l]).reshape(1, T, w.H, w.D)
                v = to_bf16_bits(h @ w.Wv[l]).reshape(1, T, w.H, w.D)
                sk[r - 1, l], sv[r - 1, l] = k, v
                out, _ = self.o.attention(self.K, self.V, l, r, r, np.array([self.P], np.int32),
                                          np.array([T], np.int32), q, k, v)
                if self.bf16_outputs:
                    out = bf16_bits_to_f64(to_bf16_bits(out))
                h = h + np.tanh(out[0].reshape(T, w.H * w.D) @ w.Wo[l])
        return (h @ w.U).astype(np.float32), sk, sv

    def commit(self, sk, sv, accepted):
        self.K, self.V, pl, flag = self.o.kv_append(self.K, self.V, sk, sv,
                                                    np.array([accepted], np.int32),
                                                    np.array([self.P], np.int32))
        assert flag == 0
        self.P = int(pl[0])

    def accept(self, logits, draft):
        acc, tid, nxt = self.o.greedy_accept(logits[None], np.asarray(draft, np.int32)[None])
        return int(acc[0]), tid[0], int(nxt[0])


class ToyLoopedGPU:
    def __init__(self, w, cap):
        import torch

        import paper_2609_34538_gb300 as das
        self.t, self.das, self.w, self.cap = torch, das, w, cap
        f = lambda a: torch.tensor(a, dtype=torch.float64, device="cuda")
        self.E, self.Wq, self.Wk, self.Wv, self.Wo, self.U = map(
            f, (w.E, w.Wq, w.Wk, w.Wv, w.Wo, w.U))
        self.cache = das.DepthKVCache.empty(w.R, w.L, 1, cap, w.H, w.D)
        self.cache.k.zero_()
        self.cache.v.zero_()
        self.pl = torch.zeros(1, dtype=torch.int32, device="cuda")
        self.flag = torch.zeros(1, dtype=torch.int32, device="cuda")
        self.ws = {}

    def forward(self, tokens):
        t, w, das = self.t, self.w, self.das
        T = len(tokens)
        if T not in self.ws:
            self.ws[T] = das.new_workspace(self.cache, w.H, T)
        h = self.E[t.tensor(list(tokens), device="cuda")]
        bl = t.full((1,), T, dtype=t.int32, device="cuda")
        sk = t.empty((w.R, w.L, 1, T, w.H, w.D), dtype=t.bfloat16, device="cuda")
        sv = t.empty_like(sk)
        for r in range(1, w.R + 1):
            for l in range(w.L):
                # fp64 -> fp32 -> bf16, the rounding path of the CPU model
                bf = lambda x: x.float().to(t.bfloat16).view(1, T, w.H, w.D)
                q = bf(h @ self.Wq[l])
                sk[r - 1, l] = bf(h @ self.Wk[l])
                sv[r - 1, l] = bf(h @ self.Wv[l])
                out, _ = das.das_verify_attention(self.cache, l, r, self.pl, bl, q, sk[r - 1, l],
                                                  sv[r - 1, l], self.ws[T])
                h = h + t.tanh(out.double().view(T, w.H * w.D) @ self.Wo[l])
        return (h @ self.U).float().contiguous(), sk, sv

    def accept(self, logits, draft):
        t = self.t
        acc, tid, nxt = self.das.das_greedy_accept(
            logits[None], t.tensor([list(draft)], dtype=t.int32, device="cuda"))
        return int(acc[0]), tid[0].cpu().numpy(), int(nxt[0])

    def commit(self, sk, sv, accepted):
        t = self.t
        acc = t.tensor([accepted], dtype=t.int32, device="cuda")
        self.das.das_kv_append(self.cache, sk, sv, acc, self.pl, self.flag)
        assert int(self.flag.item()) == 0

    @property
    def P(self):
        return int(self.pl.item())


def prefill(m, prompt):
    """Commit prompt[:-1] as one verified block; the last token is the anchor."""
    if len(prompt) > 1:
        _, sk, sv = m.forward(prompt[:-1])
        m.commit(sk, sv, len(prompt) - 1)  # all materialized: n = min(a + 1, w) = w
    return prompt[-1]


def ar(m, prompt, n, margins=None, logits_out=None):
    """Greedy AR decoding; if `margins` is a list, the gap between the two
    largest logits of every step is appended to it; if `logits_out` is a
    list, every step's logits (float64) are."""
    anchor, out = prefill(m, prompt), []
    while len(out) < n:
        logits, sk, sv = m.forward([anchor])
        a, tid, nxt = m.accept(logits, [-1])  # no proposal: the target argmax
        m.commit(sk, sv, 0)                   # the anchor is materialized
        out.append(int(tid[0]))
        anchor = out[-1]
        row = np.asarray(logits[0].cpu() if hasattr(logits, "cpu") else logits[0],
                         dtype=np.float64)
        if margins is not None:
            srt = np.sort(row)
            margins.append(srt[-1] - srt[-2])
        if logits_out is not None:
            logits_out.append(row)
    return out


def spec(m, prompt, n, propose, w):
    """propose(emitted, w) -> w proposal ids.  Returns (emitted, acceptances)."""
    anchor, out, accs = prefill(m, prompt), [], []
    while len(out) < n:
        ys = list(propose(out, w))
        logits, sk, sv = m.forward([anchor] + ys[:-1])
        a, tid, nxt = m.accept(logits, ys)
        m.commit(sk, sv, a)          # n = min(a + 1, w) inputs materialized
        out += ys[:a] + ([nxt] if a < w else [])
        anchor = nxt
        accs.append(a)
    return out[:n], accs
