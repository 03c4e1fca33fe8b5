"""Seeded synthetic inputs for the verifier: logit rows, emitted-token ids,
ragged request layouts (CSR offsets), decode traces and scorer weights.

This module is shared by the GPU tests, the benchmark and the oracle tests.  It
holds none of the verifier's arithmetic: it only draws random numbers.  The
paper evaluates on 15 benchmark suites whose model outputs are not available
here; these generators stand in for the small model's per-token distributions
with the shapes and value mixes listed below.

Workloads (vocabulary widths are the small model's output widths):

  tiny    8 requests, T ~ U{16..64}, V = 32,000 float32, x = 2 N(0,1) plus one
          spike +U(0,8) per row at a random index.
  full    64 requests, T ~ U{32..256}, V = 151,936 bfloat16, x = s N(0,1) with a
          per-row scale s ~ U(1,4); 70% of rows get a spike +U(0,12).
  decode  256 live slots for 1,000 steps, request lengths ~ U{64..1000}, a slot is
          refilled by a new request when its request ends; rows as in ``full``.
  ragged  1,024 requests, T = clip(round(lognormal(ln 128, 0.8)), 8, 1024),
          rows as in ``full``, processed in 8,192-row chunks.
  wide    512 requests, T ~ U{64..512}, V = 262,144 float32, x = 2 t_3 (Student-t,
          3 degrees of freedom); on 10% of rows the maximum is copied to a second
          random index (an exact tie for the top token).

Every row is a pure function of (workload seed, global row index): rows are
drawn in blocks of ``BLOCK`` rows from a generator seeded by the block index,
so any chunking of the batch sees identical values.  The emitted token is
sampled from the softmax of the *stored* (rounded) row at temperature 1 with
the Gumbel-max construction, which needs no normalisation.

Scorer: w (11 weights) then b are 12 draws of N(0, 0.1^2) from PCG64(seed+100),
rounded to float32; tau = 0.5.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

BLOCK = 256  # rows per seeded generation block


@dataclass
class Workload:
    name: str
    dtype: str  # "bf16" | "f32"
    vocab: int
    lengths: np.ndarray  # int64 [n_req]
    seed_host: int
    seed_dev: int
    dist: str  # "tiny" | "full" | "wide"
    chunk_rows: int = 0  # 0: whole batch in one call
    w: np.ndarray = field(default=None)  # float32 [11]
    b: float = 0.0
    tau: float = 0.5

    @property
    def n_req(self) -> int:
        return int(self.lengths.size)

    @property
    def offsets(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.lengths)]).astype(np.int64)

    @property
    def n_rows(self) -> int:
        return int(self.lengths.sum())

    @property
    def elem_bytes(self) -> int:
        return 2 if self.dtype == "bf16" else 4

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32


def scorer(seed_host: int):
    g = np.random.Generator(np.random.PCG64(seed_host + 100))
    d = g.normal(0.0, 0.1, size=12).astype(np.float32)
    return d[:11].copy(), float(d[11])


def _finish(wl: Workload) -> Workload:
    wl.w, wl.b = scorer(wl.seed_host)
    return wl


def make(name: str, n_req: int | None = None, vocab: int | None = None,
         max_len: int | None = None) -> Workload:
    """One of the five named workloads; ``n_req``/``vocab``/``max_len`` shrink it
    (same distributions) for tests that must finish quickly on the oracle."""
    if name == "tiny":
        g = np.random.Generator(np.random.PCG64(1001))
        n = n_req or 8
        lengths = g.integers(16, 64, size=n, endpoint=True)
        wl = Workload(name, "f32", vocab or 32000, lengths, 1001, 2001, "tiny")
    elif name == "full":
        g = np.random.Generator(np.random.PCG64(1002))
        n = n_req or 64
        lengths = g.integers(32, 256, size=n, endpoint=True)
        wl = Workload(name, "bf16", vocab or 151936, lengths, 1002, 2002, "full")
    elif name == "ragged":
        g = np.random.Generator(np.random.PCG64(1004))
        n = n_req or 1024
        raw = np.exp(g.normal(np.log(128.0), 0.8, size=n))
        lengths = np.clip(np.round(raw), 8, 1024).astype(np.int64)
        wl = Workload(name, "bf16", vocab or 151936, lengths, 1004, 2004, "full",
                      chunk_rows=8192)
    elif name == "wide":
        g = np.random.Generator(np.random.PCG64(1005))
        n = n_req or 512
        lengths = g.integers(64, 512, size=n, endpoint=True)
        wl = Workload(name, "f32", vocab or 262144, lengths, 1005, 2005, "wide")
    else:
        raise KeyError(name)
    wl.lengths = np.asarray(wl.lengths, np.int64)
    if max_len is not None:
        wl.lengths = np.minimum(wl.lengths, max_len)
    return _finish(wl)


# ---- rows ------------------------------------------------------------------

def _block(wl: Workload, blk: int, device) -> tuple[torch.Tensor, torch.Tensor]:
    """Rows [blk*BLOCK, (blk+1)*BLOCK) in storage dtype, and their emitted ids."""
    dev = torch.device(device)
    gen = torch.Generator(device=dev)
    gen.manual_seed(wl.seed_dev * 1_000_003 + blk)
    n, V = BLOCK, wl.vocab
    rows = torch.arange(n, device=dev)
    if wl.dist == "tiny":
        x = torch.randn(n, V, generator=gen, device=dev) * 2.0
        pos = torch.randint(0, V, (n,), generator=gen, device=dev)
        amp = torch.rand(n, generator=gen, device=dev) * 8.0
        x[rows, pos] += amp
    elif wl.dist == "full":
        s = 1.0 + 3.0 * torch.rand(n, 1, generator=gen, device=dev)
        x = torch.randn(n, V, generator=gen, device=dev) * s
        pos = torch.randint(0, V, (n,), generator=gen, device=dev)
        amp = torch.rand(n, generator=gen, device=dev) * 12.0
        has = torch.rand(n, generator=gen, device=dev) < 0.7
        x[rows, pos] += torch.where(has, amp, torch.zeros_like(amp))
    elif wl.dist == "wide":
        z = torch.randn(n, V, generator=gen, device=dev)
        c = torch.zeros(n, V, device=dev)
        for _ in range(3):
            c += torch.randn(n, V, generator=gen, device=dev).square_()
        x = 2.0 * z / torch.sqrt(c / 3.0)
        del z, c
        tie = torch.rand(n, generator=gen, device=dev) < 0.10
        other = torch.randint(0, V - 1, (n,), generator=gen, device=dev)
        top = torch.argmax(x, dim=1)
        other = other + (other >= top).long()  # a second index, never the top one
        r = rows[tie]
        x[r, other[tie]] = x[r, top[tie]]
    else:
        raise KeyError(wl.dist)
    xs = x.to(wl.torch_dtype)
    del x
    # emitted token ~ softmax(stored row) at T = 1, via Gumbel-max
    u = torch.rand(n, V, generator=gen, device=dev).clamp_(min=1e-30)
    g = -torch.log(-torch.log(u))
    chosen = torch.argmax(xs.float() + g, dim=1).to(torch.int32)
    return xs, chosen


def rows(wl: Workload, lo: int, hi: int, device="cuda", out: torch.Tensor | None = None,
         chosen_out: torch.Tensor | None = None):
    """Global rows [lo, hi) of the workload: (logits [hi-lo, V], chosen [hi-lo])."""
    n = hi - lo
    if out is None:
        out = torch.empty(n, wl.vocab, dtype=wl.torch_dtype, device=device)
    if chosen_out is None:
        chosen_out = torch.empty(n, dtype=torch.int32, device=device)
    b0, b1 = lo // BLOCK, (hi - 1) // BLOCK if n > 0 else -1
    for blk in range(b0, b1 + 1):
        x, c = _block(wl, blk, device)
        s = max(lo, blk * BLOCK)
        e = min(hi, (blk + 1) * BLOCK)
        out[s - lo:e - lo].copy_(x[s - blk * BLOCK:e - blk * BLOCK])
        chosen_out[s - lo:e - lo].copy_(c[s - blk * BLOCK:e - blk * BLOCK])
        del x, c
    return out, chosen_out


def to_oracle_array(t: torch.Tensor) -> np.ndarray:
    """Host copy in the oracle's input format: float32, or uint16 bit patterns for bf16."""
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


# ---- decode traces -----------------------------------------------------------

@dataclass
class DecodeTrace:
    n_slots: int
    n_steps: int
    vocab: int
    dtype: str
    seed_dev: int
    dist: str
    requests: list  # (slot, start_step, length) for every request that started
    eos: np.ndarray  # uint8 [n_steps, n_slots]
    w: np.ndarray
    b: float
    tau: float = 0.5

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32

    def as_workload(self) -> Workload:
        """Row generator view: global row id = step * n_slots + slot."""
        wl = Workload("decode", self.dtype, self.vocab, np.zeros(0, np.int64), 1003,
                      self.seed_dev, self.dist)
        wl.w, wl.b, wl.tau = self.w, self.b, self.tau
        return wl


def decode_trace(n_slots: int = 256, n_steps: int = 1000, lo: int = 64, hi: int = 1000,
                 vocab: int = 151936, seed_host: int = 1003, seed_dev: int = 2003) -> DecodeTrace:
    """Every slot is always live: when a request ends the slot takes a new one."""
    g = np.random.Generator(np.random.PCG64(seed_host))
    eos = np.zeros((n_steps, n_slots), np.uint8)
    reqs = []
    for s in range(n_slots):
        t = 0
        while t < n_steps:
            L = int(g.integers(lo, hi, endpoint=True))
            reqs.append((s, t, L))
            if t + L - 1 < n_steps:
                eos[t + L - 1, s] = 1
            t += L
    w, b = scorer(seed_host)
    return DecodeTrace(n_slots, n_steps, vocab, "bf16", seed_dev, "full", reqs, eos, w, b)


# ---- scorer head weights ---------------------------------------------------------

HEAD_D, HEAD_HEADS, HEAD_DFF, HEAD_DIN = 64, 4, 128, 4


def head_param_count(n_layers: int) -> int:
    per_layer = (3 * HEAD_D * HEAD_D + 3 * HEAD_D + HEAD_D * HEAD_D + HEAD_D + 2 * HEAD_D
                 + HEAD_DFF * HEAD_D + HEAD_DFF + HEAD_D * HEAD_DFF + HEAD_D + 2 * HEAD_D)
    return HEAD_D * HEAD_DIN + HEAD_D + n_layers * per_layer + HEAD_D + 1


def head_weights(n_layers: int = 2, seed: int = 3001) -> np.ndarray:
    """Seeded stand-in for the head's trained weights (flat float32, the layout
    the library documents): matrices N(0, 1/fan_in), biases N(0, 0.02^2),
    LayerNorm gains 1 + N(0, 0.1^2) and shifts N(0, 0.1^2)."""
    g = np.random.Generator(np.random.PCG64(seed))
    D, F, I = HEAD_D, HEAD_DFF, HEAD_DIN
    parts = []

    def mat(rows, cols):
        parts.append(g.normal(0.0, 1.0 / np.sqrt(cols), size=rows * cols))

    def vec(n, scale=0.02, base=0.0):
        parts.append(base + g.normal(0.0, scale, size=n))

    mat(D, I)
    vec(D)
    for _ in range(n_layers):
        mat(3 * D, D)
        vec(3 * D)
        mat(D, D)
        vec(D)
        vec(D, 0.1, 1.0)
        vec(D, 0.1)
        mat(F, D)
        vec(F)
        mat(D, F)
        vec(D)
        vec(D, 0.1, 1.0)
        vec(D, 0.1)
    mat(1, D)
    vec(1)
    w = np.concatenate(parts).astype(np.float32)
    assert w.size == head_param_count(n_layers)
    return w


def head_features(lengths, seed: int = 4001) -> tuple[np.ndarray, np.ndarray]:
    """Seeded row records for the scorer head: (feat float32 [n_rows][8], offsets).

    Slot values follow the verifier's record layout: m ~ U(0.02, 1); the
    emitted token is the top one on half of the rows (l = log m), otherwise
    l = log m - Exp(mean 2); h ~ -U(0, ln 20); rho = t / T with t 1-based.  The
    slots the head does not read (margin, entropy, LSE, x1) hold N(0, 5^2)
    noise so that reading a wrong slot shows up.
    """
    lengths = np.asarray(lengths, np.int64)
    offsets = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    n = int(offsets[-1])
    g = np.random.Generator(np.random.PCG64(seed))
    feat = g.normal(0.0, 5.0, size=(n, 8))
    m = g.uniform(0.02, 1.0, size=n)
    top = g.random(n) < 0.5
    feat[:, 0] = np.log(m) - np.where(top, 0.0, g.exponential(2.0, size=n))
    feat[:, 1] = m
    feat[:, 4] = -g.uniform(0.0, np.log(20.0), size=n)
    for r in range(lengths.size):
        T = int(lengths[r])
        feat[offsets[r]:offsets[r + 1], 5] = np.arange(1, T + 1) / max(T, 1)
    return feat.astype(np.float32), offsets


# ---- validation pools for calibration -----------------------------------------------------

def selective_pool(n: int, seed: int = 5001, nan_frac: float = 0.01):
    """Seeded stand-in for a validation pool of verifier outputs:
    (scores float32 [n], labels uint8 [n]).  z ~ N(0, 1.5^2), score =
    sigmoid(z) rounded to float32 (so equal scores occur as they do in a real
    pool), label = 1 (correct) with probability equal to the score, and a
    fraction `nan_frac` of requests flagged (score NaN)."""
    g = np.random.Generator(np.random.PCG64(seed))
    z = g.normal(0.0, 1.5, size=n)
    s = (1.0 / (1.0 + np.exp(-z))).astype(np.float32)
    y = (g.random(n) < s).astype(np.uint8)
    s[g.random(n) < nan_frac] = np.float32(np.nan)
    return s, y


# ---- quantile-summary + MLP aggregator weights --------------------------------------------

QMLP_NS, QMLP_H = 28, 64


def qmlp_param_count() -> int:
    return QMLP_H * QMLP_NS + QMLP_H + QMLP_H * QMLP_H + QMLP_H + QMLP_H + 1


def qmlp_weights(seed: int = 6001) -> np.ndarray:
    """Seeded stand-in for the quantile-summary MLP's trained weights (flat
    float32 in the library's layout): matrices N(0, 1/fan_in), biases
    N(0, 0.02^2)."""
    g = np.random.Generator(np.random.PCG64(seed))
    parts = [g.normal(0.0, 1.0 / np.sqrt(QMLP_NS), QMLP_H * QMLP_NS), g.normal(0.0, 0.02, QMLP_H),
             g.normal(0.0, 1.0 / np.sqrt(QMLP_H), QMLP_H * QMLP_H), g.normal(0.0, 0.02, QMLP_H),
             g.normal(0.0, 1.0 / np.sqrt(QMLP_H), QMLP_H), g.normal(0.0, 0.02, 1)]
    w = np.concatenate(parts).astype(np.float32)
    assert w.size == qmlp_param_count()
    return w


# ---- LM-head inputs --------------------------------------------------------------------

def lmhead_inputs(n_rows: int, d: int = 3584, vocab: int = 151936, seed: int = 8001,
                  device="cuda"):
    """Seeded stand-ins for the small model's final hidden states and LM head
    (trained weights are not available): hidden bf16 [n_rows][d] with N(0, 1)
    entries and a per-row scale U(0.5, 2); weight bf16 [vocab][d] with
    N(0, (2 / sqrt(d))^2) entries, so the logits have a scale of a few units;
    emitted token ids uniform in [0, vocab).  d = 3,584 is the hidden size the
    paper quotes for the small model (Table 2)."""
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    h = torch.randn(n_rows, d, generator=g, device=dev)
    h *= 0.5 + 1.5 * torch.rand(n_rows, 1, generator=g, device=dev)
    hidden = h.to(torch.bfloat16)
    del h
    weight = torch.empty(vocab, d, dtype=torch.bfloat16, device=dev)
    step = 8192
    for v0 in range(0, vocab, step):  # in slices: no fp32 copy of the whole matrix
        v1 = min(vocab, v0 + step)
        weight[v0:v1] = (torch.randn(v1 - v0, d, generator=g, device=dev) *
                         (2.0 / d ** 0.5)).to(torch.bfloat16)
    chosen = torch.randint(0, vocab, (n_rows,), generator=g, device=dev, dtype=torch.int32)
    return hidden, weight, chosen


# ---- prompts for the pre-scorer (Section 3.1, Eq. 2) --------------------------------------
#
# The paper's prompts (benchmark questions with images) are not available;
# these stand in for them: a seeded vocabulary of VOCAB pseudo-words (random
# lowercase strings of 3-10 letters), words drawn with Zipf(1.07) frequencies
# over the vocabulary's ranks, prompt lengths clip(round(lognormal(ln 30,
# 0.7)), 3, 400) words, about 10% of words capitalised, punctuation after 10%
# of words, a number token for 3%, a one-letter word (which no token keeps)
# for 5%, a word with a non-ASCII letter for 1%; image counts 0 (30%), 1
# (55%), 2 (10%) or 3-5 (5%).

PROMPT_VOCAB = 20000


def _pseudo_words(n: int, seed: int) -> list[bytes]:
    """n distinct random lowercase words of 3-10 letters (a drawn length is
    raised by one after every eight collisions, so the loop always ends)."""
    g = np.random.Generator(np.random.PCG64(seed))
    lens = g.integers(3, 10, size=n, endpoint=True)
    letters = np.frombuffer(b"abcdefghijklmnopqrstuvwxyz", np.uint8)
    words, seen = [], set()
    for L in lens:
        tries = 0
        while True:
            w = bytes(letters[g.integers(0, 26, size=int(L) + tries // 8)])
            if w not in seen:
                seen.add(w)
                words.append(w)
                break
            tries += 1
    return words


def prompts(n: int, seed: int = 9001) -> tuple[list[bytes], np.ndarray]:
    """n seeded synthetic prompts (UTF-8 bytes) and their image counts."""
    words = _pseudo_words(PROMPT_VOCAB, seed + 1)
    ranks = np.arange(1, PROMPT_VOCAB + 1, dtype=np.float64)
    pz = ranks ** -1.07
    pz /= pz.sum()
    g = np.random.Generator(np.random.PCG64(seed))
    lengths = np.clip(np.round(np.exp(g.normal(np.log(30.0), 0.7, size=n))), 3, 400).astype(int)
    out = []
    for L in lengths:
        idx = g.choice(PROMPT_VOCAB, size=L, p=pz)
        u = g.random((L, 6))
        parts = []
        for k in range(L):
            w = words[idx[k]]
            if u[k, 0] < 0.10:
                w = w[:1].upper() + w[1:]
            if u[k, 1] < 0.03:
                w = b"%d" % int(u[k, 2] * 1000)
            elif u[k, 1] < 0.08:
                w = w[:1]
            elif u[k, 1] < 0.09:
                w = w + "é".encode()
            if u[k, 3] < 0.10:
                w = w + b".,?!:;"[int(u[k, 4] * 6):][:1]
            parts.append(w)
        out.append(b" ".join(parts))
    c = g.random(n)
    images = np.where(c < 0.30, 0, np.where(c < 0.85, 1, np.where(c < 0.95, 2,
                                                                   3 + (c * 1000).astype(int) % 3)))
    return out, images.astype(np.int32)


def prescore_weights(vocab: int, seed: int = 9101) -> tuple[np.ndarray, float]:
    """Stand-in weights of the pre-scorer's logistic regression (the trained
    ones are not available): V TF-IDF weights N(0, 1), the image-count weight
    N(0, 0.3^2), the length weight N(0, 0.01^2), then b ~ N(0, 0.1^2)."""
    g = np.random.Generator(np.random.PCG64(seed))
    w = np.concatenate([g.normal(0.0, 1.0, vocab), g.normal(0.0, 0.3, 1),
                        g.normal(0.0, 0.01, 1)]).astype(np.float32)
    return w, float(g.normal(0.0, 0.1))
