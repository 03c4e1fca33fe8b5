"""Float64 oracle of the prompt pre-scorer (Pro-Router, Section 3.1, Eq. 2).

Test infrastructure only: tests, the package's smoke check and the bench's
CPU-baseline leg use it; the library never does.

    p_pre(x) = sigmoid(w . phi(x) + b)

with phi(x) the concatenation of the prompt text's TF-IDF vector, the image
count and the prompt length (Section 3.1).  The paper names the features and
the logistic regression but not the TF-IDF variant or the tokenizer; the
readings (also listed in the design notes):
  * tokens: maximal runs of word bytes ([0-9A-Za-z_] and every byte >= 0x80)
    at least two bytes long, after lowercasing ASCII letters -- on ASCII text
    the usual default of TF-IDF vectorizers (two or more word characters);
  * vocabulary: every term of the fitting corpus with document frequency
    >= min_df, columns in byte order of the terms;
  * tf = raw count in the prompt; idf = ln((1 + n) / (1 + df)) + 1 (smoothed);
    the row tf * idf scaled to unit Euclidean length (a row with no
    vocabulary term stays zero);
  * prompt length = the number of tokens of the prompt (in or out of the
    vocabulary); image count as given;
  * w has V + 2 entries: V TF-IDF weights, then the image-count weight, then
    the length weight.
Everything in float64, sums in ascending column order.
"""
from __future__ import annotations

import math
import re

_TOKEN = re.compile(rb"[0-9A-Za-z_\x80-\xff]{2,}")


def tokens(text: bytes) -> list[bytes]:
    """The prompt's tokens, ASCII letters lowercased (bytes.lower touches only ASCII)."""
    return _TOKEN.findall(text.lower())


class Model:
    def __init__(self, terms: list[bytes], idf: list[float], n_docs: int):
        self.terms = terms
        self.idf = idf
        self.n_docs = n_docs
        self.index = {t: j for j, t in enumerate(terms)}


def fit(docs: list[bytes], min_df: int = 1) -> Model:
    """Vocabulary and smoothed idf of a corpus."""
    df: dict[bytes, int] = {}
    for d in docs:
        for t in set(tokens(d)):
            df[t] = df.get(t, 0) + 1
    terms = sorted(t for t, c in df.items() if c >= min_df)
    n = len(docs)
    idf = [math.log((1.0 + n) / (1.0 + df[t])) + 1.0 for t in terms]
    return Model(terms, idf, n)


def features(model: Model, prompt: bytes, n_images: int):
    """phi(x): the TF-IDF row as {column: value} (unit length or empty), the
    image count and the prompt length."""
    toks = tokens(prompt)
    counts: dict[int, int] = {}
    for t in toks:
        j = model.index.get(t)
        if j is not None:
            counts[j] = counts.get(j, 0) + 1
    row = {j: c * model.idf[j] for j, c in counts.items()}
    norm = math.sqrt(sum(v * v for _, v in sorted(row.items())))
    if norm > 0.0:
        row = {j: v / norm for j, v in row.items()}
    return row, float(n_images), float(len(toks))


def logit(model: Model, prompt: bytes, n_images: int, w, b: float) -> float:
    """z = w . phi(x) + b (Eq. 2 before the sigmoid)."""
    row, img, length = features(model, prompt, n_images)
    V = len(model.terms)
    z = float(b)
    for j in sorted(row):
        z += float(w[j]) * row[j]
    z += float(w[V]) * img + float(w[V + 1]) * length
    return z


def score(model: Model, prompts: list[bytes], n_images, w, b: float):
    """(p_pre, z) for every prompt."""
    zs = [logit(model, p, int(k), w, b) for p, k in zip(prompts, n_images)]
    ps = [1.0 / (1.0 + math.exp(-z)) if z >= 0 else math.exp(z) / (1.0 + math.exp(z)) for z in zs]
    return ps, zs
