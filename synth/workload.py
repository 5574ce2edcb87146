"""Seeded synthetic workloads shaped like the paper's decoding steps.

A workload is one denoising step of a batch: partial outputs x (token ids,
-1 = MASK), the proposed positions, K candidate tokens per position with fp32
confidences, and the vocabulary as byte strings.  Construction:

1. sample a length-steered random derivation of the grammar and render every
   terminal as a sample lexeme (space-separated when the grammar has a
   skipped whitespace terminal, concatenated otherwise);
2. tokenize the text greedily (longest vocabulary match);
3. pad the tail with MASK to n tokens and mask uniformly at the stated rate;
4. propose k masked positions uniformly; draw K distinct candidates per
   position by Gumbel-top-K over N(0,1) fp32 logits, the true (witness) token's
   logit raised by ln|vocab| + 1 so that it is usually among them;
5. confidence = the candidate's softmax probability (fp32).

No step here lexes, parses or decides validity: the data are produced from
the grammar's render recipes alone.
"""
from __future__ import annotations

import heapq
from dataclasses import dataclass
import numpy as np

from .grammars import GrammarSpec, grammar_for


@dataclass
class WorkloadSpec:
    name: str
    batch: int
    n: int
    mask_rate: float
    k: int
    K: int
    vocab: int
    tok_len: tuple          # (lo, hi)
    zipf: float | None      # None = uniform lengths
    uniform_cands: bool = False


WORKLOADS = {
    'expr-tiny': WorkloadSpec('expr-tiny', 1, 32, 0.25, 8, 8, 256, (1, 3), None, True),
    'json-schema': WorkloadSpec('json-schema', 16, 256, 0.40, 4, 16, 32768, (1, 8), 1.2),
    'clike-512': WorkloadSpec('clike-512', 32, 512, 0.50, 8, 32, 65536, (1, 10), 1.2),
    'random-stress-1024': WorkloadSpec('random-stress-1024', 64, 1024, 0.60, 16, 32, 126000,
                                       (1, 10), 1.2),
    'smiles-256': WorkloadSpec('smiles-256', 256, 256, 0.50, 16, 16, 126000, (1, 10), 1.2),
}


@dataclass
class Workload:
    name: str
    seed: int
    grammar: GrammarSpec
    vocab: list             # list[bytes]
    x: np.ndarray           # int32 [B][n], -1 = MASK
    witness: np.ndarray     # int32 [B][n], the sentence's tokens (-1 past its end)
    pos: np.ndarray         # int32 [B][k]
    cand: np.ndarray        # int32 [B][k][K]
    conf: np.ndarray        # float32 [B][k][K]

    @property
    def B(self):
        return self.x.shape[0]

    @property
    def n(self):
        return self.x.shape[1]

    @property
    def k(self):
        return self.pos.shape[1]

    @property
    def K(self):
        return self.cand.shape[2]

    def vocab_arrays(self):
        """(tok_off int32 [V+1], tok_bytes uint8) -- the C-ABI vocab layout."""
        lens = np.fromiter((len(t) for t in self.vocab), np.int64, len(self.vocab))
        off = np.zeros(len(self.vocab) + 1, np.int32)
        off[1:] = np.cumsum(lens)
        data = np.frombuffer(b''.join(self.vocab), np.uint8).copy()
        return off, data


# ---------------------------------------------------------------- derivations

def _min_yield(g: GrammarSpec):
    """Minimal number of terminals each nonterminal derives, and the production
    that attains it, settled in increasing cost (well-founded choice)."""
    T = g.T
    INF = 1 << 60
    cost = [INF] * g.V
    best = [-1] * g.V
    users = [[] for _ in range(g.V)]
    missing = []
    for pi, (lhs, rhs) in enumerate(g.productions):
        nts = [s - T for s in rhs if s >= T]
        missing.append(len(nts))
        for a in nts:
            users[a].append(pi)
    heap = []
    for pi, (lhs, rhs) in enumerate(g.productions):
        if missing[pi] == 0:
            heapq.heappush(heap, (len(rhs), pi))
    settled = [False] * g.V
    while heap:
        c, pi = heapq.heappop(heap)
        a = g.productions[pi][0]
        if settled[a]:
            continue
        settled[a] = True
        cost[a] = c
        best[a] = pi
        for u in users[a]:
            missing[u] -= 1
            if missing[u] == 0:
                rhs = g.productions[u][1]
                cu = sum(1 if s < T else cost[s - T] for s in rhs)
                heapq.heappush(heap, (cu, u))
    if not all(settled):
        raise ValueError('grammar has unproductive nonterminals')
    return cost, best


def sample_derivation(g: GrammarSpec, rng, target: int):
    """Leftmost derivation steered towards about `target` terminals."""
    T = g.T
    cost, best = _min_yield(g)
    by_lhs = [[] for _ in range(g.V)]
    for pi, (lhs, rhs) in enumerate(g.productions):
        by_lhs[lhs].append(pi)
    pcost = [sum(1 if s < T else cost[s - T] for s in rhs) for _, rhs in g.productions]
    out = []
    stack = [T + g.start]
    committed = cost[g.start]
    while stack:
        s = stack.pop()
        if s < T:
            out.append(s)
            continue
        a = s - T
        if committed >= target:
            pi = best[a]
        else:
            cands = by_lhs[a]
            room = target - committed
            ok = [p for p in cands if pcost[p] - cost[a] <= room]
            if not ok:
                pi = best[a]
            else:
                w = np.array([1.0 + (pcost[p] - cost[a]) for p in ok])
                pi = ok[int(rng.choice(len(ok), p=w / w.sum()))]
        committed += pcost[pi] - cost[a]
        stack.extend(reversed(g.productions[pi][1]))
    return out


def _render_terminal(term, rng, reserved):
    r = term.render
    kind = r[0]
    for _ in range(100):
        if kind == 'lit':
            return r[1]
        if kind == 'lit_choice':
            return r[1][int(rng.integers(len(r[1])))]
        if kind == 'ws':
            return ' '
        if kind == 'digits':
            L = int(rng.integers(r[1], r[2] + 1))
            s = ''.join(str(int(d)) for d in rng.integers(0, 10, L))
        elif kind == 'word':
            L = int(rng.integers(r[3], r[4] + 1))
            s = r[1][int(rng.integers(len(r[1])))] + ''.join(
                r[2][int(i)] for i in rng.integers(0, len(r[2]), L - 1))
        elif kind == 'string':
            L = int(rng.integers(r[2], r[3] + 1))
            s = '"' + ''.join(r[1][int(i)] for i in rng.integers(0, len(r[1]), L)) + '"'
        elif kind == 'number':
            s = '-' if rng.random() < 0.2 else ''
            if rng.random() < 0.2:
                s += '0'
            else:
                s += str(int(rng.integers(1, 10))) + ''.join(
                    str(int(d)) for d in rng.integers(0, 10, int(rng.integers(0, 4))))
            if rng.random() < 0.3:
                s += '.' + ''.join(str(int(d)) for d in rng.integers(0, 10, int(rng.integers(1, 4))))
            if rng.random() < 0.1:
                s += 'e' + ('-' if rng.random() < 0.5 else '') + str(int(rng.integers(0, 40)))
        elif kind == 'number_simple':
            s = ''.join(str(int(d)) for d in rng.integers(0, 10, int(rng.integers(1, 5))))
            if rng.random() < 0.2:
                s += '.' + ''.join(str(int(d)) for d in rng.integers(0, 10, int(rng.integers(1, 3))))
        else:
            raise ValueError(kind)
        if s not in reserved:
            return s
    raise RuntimeError('could not render ' + term.name)


def render(g: GrammarSpec, terms, rng) -> str:
    sep = ' ' if g.has_ws else ''
    return sep.join(_render_terminal(g.terminals[t], rng, g.reserved) for t in terms)


# ------------------------------------------------------------------- vocab

def _lengths(rng, n, lo, hi, zipf):
    ls = np.arange(lo, hi + 1)
    if zipf is None:
        p = np.full(len(ls), 1.0 / len(ls))
    else:
        p = ls.astype(np.float64) ** (-zipf)
        p /= p.sum()
    return rng.choice(ls, size=n, p=p)


def make_vocab(g: GrammarSpec, spec: WorkloadSpec, rng, samples):
    """All single characters of the text, then substrings of sample renderings
    and random strings over the charset (half each), lengths per the spec."""
    chars = sorted(set(g.charset) | set(''.join(samples)))
    vocab = list(dict.fromkeys(chars))
    seen = set(vocab)
    text = '\x00'.join(samples)
    want = spec.vocab
    tries = 0
    while len(vocab) < want:
        m = min(8192, 2 * (want - len(vocab)) + 16)
        Ls = _lengths(rng, m, spec.tok_len[0], spec.tok_len[1], spec.zipf)
        src = rng.random(m) < 0.5
        starts = rng.integers(0, max(1, len(text) - 12), m)
        for L, from_text, st in zip(Ls, src, starts):
            if from_text:
                s = text[st:st + L]
                if '\x00' in s or len(s) != L:
                    continue
            else:
                s = ''.join(chars[int(i)] for i in rng.integers(0, len(chars), L))
            if s not in seen:
                seen.add(s)
                vocab.append(s)
                if len(vocab) == want:
                    break
        tries += 1
        if tries > 10000:
            raise RuntimeError('vocab generation stalled')
    return [s.encode('latin-1') for s in vocab]


def tokenize(text: bytes, index: dict, maxlen: int):
    """Greedy longest-match tokenization (every single byte is in the vocab)."""
    out = []
    i = 0
    n = len(text)
    while i < n:
        for L in range(min(maxlen, n - i), 0, -1):
            t = index.get(text[i:i + L])
            if t is not None:
                out.append(t)
                i += L
                break
        else:
            raise ValueError('byte %r not in vocab' % text[i:i + 1])
    return out


# -------------------------------------------------------------- workloads

def _sentence_tokens(g, rng, index, maxlen, n):
    """Witness sentence tokenized to at most n tokens, filling most of n."""
    target = max(1, n // 2)
    best = None
    for _ in range(40):
        terms = sample_derivation(g, rng, target)
        text = render(g, terms, rng).encode('latin-1')
        toks = tokenize(text, index, maxlen)
        if len(toks) <= n:
            if best is None or len(toks) > len(best):
                best = toks
            if len(toks) >= int(0.8 * n):
                return toks
            target = int(target * max(1.05, min(2.0, 0.9 * n / max(1, len(toks)))))
        else:
            target = max(1, int(target * 0.85 * n / len(toks)))
    if best is None:
        raise RuntimeError('could not fit a sentence into %d tokens' % n)
    return best


def make_workload(name: str, seed: int = 42, batch: int | None = None, k: int | None = None,
                  n: int | None = None, K: int | None = None, vocab_size: int | None = None):
    """Build the named workload; optional overrides shrink it for tests."""
    spec = WORKLOADS[name]
    B = batch or spec.batch
    n = n or spec.n
    kk = k or spec.k
    KK = K or spec.K
    V = vocab_size or spec.vocab
    g = grammar_for(name)
    rng = np.random.Generator(np.random.PCG64(seed))
    samples = [render(g, sample_derivation(g, rng, 40), rng) for _ in range(64)]
    vspec = WorkloadSpec(spec.name, B, n, spec.mask_rate, kk, KK, V, spec.tok_len, spec.zipf,
                         spec.uniform_cands)
    vocab = make_vocab(g, vspec, rng, samples)
    index = {t: i for i, t in enumerate(vocab)}
    maxlen = max(len(t) for t in vocab)
    x = np.full((B, n), -1, np.int32)
    wit = np.full((B, n), -1, np.int32)
    pos = np.zeros((B, kk), np.int32)
    for b in range(B):
        toks = _sentence_tokens(g, rng, index, maxlen, n)
        m = len(toks)
        wit[b, :m] = toks
        x[b, :m] = toks
        n_mask = int(round(spec.mask_rate * n))
        extra = max(0, n_mask - (n - m))
        if extra > 0:
            idx = rng.choice(m, size=min(extra, m), replace=False)
            x[b, idx] = -1
        masked = np.flatnonzero(x[b] < 0)
        take = min(kk, len(masked))
        sel = np.sort(rng.choice(masked, size=take, replace=False))
        if take < kk:           # not enough masks: repeat is not allowed, so
            raise ValueError('workload %s: only %d masked positions' % (name, len(masked)))
        pos[b] = sel
    cand = np.zeros((B, kk, KK), np.int32)
    conf = np.zeros((B, kk, KK), np.float32)
    boost = np.float32(np.log(V) + 1.0)
    for b in range(B):
        for j in range(kk):
            p = pos[b, j]
            if spec.uniform_cands:
                logits = np.zeros(V, np.float32)
            else:
                logits = rng.standard_normal(V, dtype=np.float32)
                if wit[b, p] >= 0:
                    logits[wit[b, p]] += boost
            gum = logits - np.log(-np.log(rng.random(V, dtype=np.float32) + np.float32(1e-20))
                                  + np.float32(1e-20))
            top = np.argpartition(-gum, KK - 1)[:KK]
            top = top[np.argsort(-gum[top], kind='stable')]
            mx = logits.max()
            e = np.exp(logits - mx)
            prob = e / e.sum(dtype=np.float32)
            cand[b, j] = top
            conf[b, j] = prob[top].astype(np.float32)
    return Workload(name, seed, g, vocab, x, wit, pos, cand, conf)
