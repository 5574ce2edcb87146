"""Seeded synthetic grammars that stand in for the paper's task grammars.

The paper evaluates on C++, schema-derived JSON and SMILES grammars that come
from prior work and are not available; these generators build grammars with
the stated shapes instead (counts of nonterminals, productions, terminals,
recursion).  Nothing here implements any part of the validity check: a grammar
is data (terminal regexes, productions) plus, for each terminal, a recipe to
render a sample lexeme so that witness sentences can be produced.

Symbol numbering (shared with the C-ABI): terminals are 0..T-1, nonterminal j
is T+j.  Terminal priority is its index (lower index wins a tie).

Regex syntax understood by both the product library and the oracle (each has
its own parser): literal bytes, escapes ``\\c`` for any punctuation byte c plus
``\\n \\t \\r``, classes ``[a-z_]`` / ``[^"]`` with ranges, grouping ``( )``,
alternation ``|`` and the postfix operators ``* + ?``.
"""
from __future__ import annotations

from dataclasses import dataclass, field
import numpy as np

_SPECIAL = set('\\|()[]*+?.')
_CLASS_SPECIAL = set('\\]^-[')


def rx_lit(s: str) -> str:
    """Regex matching exactly the literal string s."""
    out = []
    for c in s:
        if c == '\n':
            out.append('\\n')
        elif c == '\t':
            out.append('\\t')
        elif c in _SPECIAL:
            out.append('\\' + c)
        else:
            out.append(c)
    return ''.join(out)


def rx_class(chars: str, negate: bool = False) -> str:
    """Regex class matching any single byte of chars (ranges compressed)."""
    cs = sorted(set(chars))
    parts = []
    i = 0
    while i < len(cs):
        j = i
        while j + 1 < len(cs) and ord(cs[j + 1]) == ord(cs[j]) + 1:
            j += 1

        def esc(c):
            if c == '\n':
                return '\\n'
            if c == '\t':
                return '\\t'
            return '\\' + c if c in _CLASS_SPECIAL else c
        if j - i >= 2:
            parts.append(esc(cs[i]) + '-' + esc(cs[j]))
        else:
            parts.extend(esc(c) for c in cs[i:j + 1])
        i = j + 1
    return '[' + ('^' if negate else '') + ''.join(parts) + ']'


LOWER = 'abcdefghijklmnopqrstuvwxyz'
UPPER = LOWER.upper()
DIGIT = '0123456789'


@dataclass
class Terminal:
    name: str
    regex: str
    skip: bool = False
    # render recipe: ('lit', s) | ('word', first, rest, lo, hi) | ('ws',)
    # | ('number',) | ('string', chars, lo, hi) | ('digits', lo, hi)
    render: tuple = ()


@dataclass
class GrammarSpec:
    name: str
    terminals: list
    nonterminals: list
    start: int                       # nonterminal index (0-based among NTs)
    productions: list                # (lhs NT index, [symbol ids])
    charset: str = ''                # bytes used by the grammar's lexemes
    has_ws: bool = True
    reserved: set = field(default_factory=set)  # literal strings a class render must avoid

    @property
    def T(self):
        return len(self.terminals)

    @property
    def V(self):
        return len(self.nonterminals)

    def sym_name(self, s):
        return self.terminals[s].name if s < self.T else self.nonterminals[s - self.T]

    def rhs_flat(self):
        lhs = np.array([p[0] for p in self.productions], np.int32)
        off = np.zeros(len(self.productions) + 1, np.int32)
        for i, p in enumerate(self.productions):
            off[i + 1] = off[i] + len(p[1])
        rhs = np.array([s for p in self.productions for s in p[1]], np.int32)
        return lhs, off, rhs


class _Builder:
    """Small helper to write grammars by symbol name."""

    def __init__(self, name):
        self.name = name
        self.terms = []
        self.tidx = {}
        self.nts = []
        self.nidx = {}
        self.prods = []

    def term(self, name, regex, render, skip=False):
        self.tidx[name] = len(self.terms)
        self.terms.append(Terminal(name, regex, skip, render))

    def lit(self, s, name=None):
        self.term(name or s, rx_lit(s), ('lit', s))

    def nt(self, name):
        if name not in self.nidx:
            self.nidx[name] = len(self.nts)
            self.nts.append(name)
        return name

    def rule(self, lhs, *alts):
        self.nt(lhs)
        for alt in alts:
            syms = alt.split() if isinstance(alt, str) else list(alt)
            self.prods.append((lhs, syms))

    def build(self, start, charset, has_ws=True, reserved=()):
        T = len(self.terms)
        for _, syms in self.prods:
            for s in syms:
                if s not in self.tidx:
                    self.nt(s)
        prods = []
        for lhs, syms in self.prods:
            ids = []
            for s in syms:
                ids.append(self.tidx[s] if s in self.tidx else T + self.nidx[s])
            prods.append((self.nidx[lhs], ids))
        return GrammarSpec(self.name, self.terms, self.nts, self.nidx[start], prods,
                           charset, has_ws, set(reserved))


def expr_grammar() -> GrammarSpec:
    """Tiny arithmetic-expression CFG: 6 nonterminals, 14 productions and 10
    single-character-class terminals (digit runs collapsed to NUM, + - * / %
    ^ ( ) and whitespace)."""
    b = _Builder('expr-tiny')
    b.term('NUM', '[0-9]+', ('digits', 1, 3))
    for c in '+-*/%^()':
        b.lit(c)
    b.term('WS', '[ ]+', ('ws',), skip=True)
    b.rule('E', 'E A T', 'T')
    b.rule('A', '+', '-')
    b.rule('T', 'T M F', 'F')
    b.rule('M', '*', '/', '%')
    b.rule('F', 'U ^ F', 'U')
    b.rule('U', '( E )', 'NUM', '- U')
    return b.build('E', DIGIT + '+-*/%^() ')


_JSON_KEYS = ['id', 'name', 'email', 'age', 'active', 'tags', 'address', 'street', 'city',
              'zip', 'country', 'phone', 'orders', 'order_id', 'items', 'sku', 'qty',
              'price', 'total', 'status', 'created', 'updated', 'notes', 'meta',
              'score', 'rank', 'owner', 'version']


def json_grammar() -> GrammarSpec:
    """Schema-derived JSON CFG with RFC 8259 structure: a root object with a
    fixed sequence of typed keys, nested objects and arrays, free-form values,
    key literals as terminals (about 25 nonterminals, 70 productions, 40
    terminals)."""
    b = _Builder('json-schema')
    for k in _JSON_KEYS:                       # key literals outrank STRING
        b.lit('"%s"' % k, 'K_' + k)
    for c in '{}[]:,':
        b.lit(c)
    for w in ('true', 'false', 'null'):
        b.lit(w)
    str_chars = LOWER + UPPER + DIGIT + ' _-.@'
    b.term('STRING', '"' + rx_class('"\\\n', negate=True) + '*"', ('string', str_chars, 0, 12))
    b.term('NUMBER', '\\-?(0|[1-9][0-9]*)(\\.[0-9]+)?([eE][\\+\\-]?[0-9]+)?', ('number',))
    b.term('WS', '[ \\n\\t]+', ('ws',), skip=True)
    K = lambda k: 'K_' + k
    b.rule('Root', '{ RootBody }')
    b.rule('RootBody', f'{K("id")} : NUMBER , {K("name")} : STRING , RootRest')
    b.rule('RootRest', 'Email , Age , Active , Tags , Address , Orders , Extra',
           'Email , Active , Tags , Address , Orders , Extra',
           'Age , Active , Tags , Address , Orders',
           'Active , Tags , Address , Orders , Extra')
    b.rule('Email', f'{K("email")} : STRING', f'{K("email")} : null')
    b.rule('Age', f'{K("age")} : NUMBER', f'{K("age")} : null')
    b.rule('Active', f'{K("active")} : Bool')
    b.rule('Bool', 'true', 'false')
    b.rule('Tags', f'{K("tags")} : [ ]', f'{K("tags")} : [ StrList ]')
    b.rule('StrList', 'STRING', 'StrList , STRING')
    b.rule('Address', f'{K("address")} : AddrObj', f'{K("address")} : null')
    b.rule('AddrObj', '{ AddrBody }')
    b.rule('AddrBody', f'{K("street")} : STRING , {K("city")} : STRING , AddrTail')
    b.rule('AddrTail', f'{K("zip")} : STRING , {K("country")} : STRING',
           f'{K("country")} : STRING', f'{K("zip")} : NUMBER , {K("country")} : STRING , Phone')
    b.rule('Phone', f'{K("phone")} : STRING', f'{K("phone")} : [ StrList ]')
    b.rule('Orders', f'{K("orders")} : [ ]', f'{K("orders")} : [ OrderList ]')
    b.rule('OrderList', 'Order', 'OrderList , Order')
    b.rule('Order', '{ OrderBody }')
    b.rule('OrderBody', f'{K("order_id")} : NUMBER , {K("items")} : [ ItemList ] , OrderTail',
           f'{K("order_id")} : STRING , {K("items")} : [ ItemList ] , OrderTail')
    b.rule('ItemList', 'Item', 'ItemList , Item')
    b.rule('Item', f'{{ {K("sku")} : STRING , {K("qty")} : NUMBER , {K("price")} : NUMBER }}',
           f'{{ {K("sku")} : STRING , {K("qty")} : NUMBER }}')
    b.rule('OrderTail', f'{K("total")} : NUMBER , {K("status")} : Status , Stamps',
           f'{K("total")} : NUMBER , {K("status")} : Status')
    b.rule('Status', 'STRING', 'null', 'NUMBER')
    b.rule('Stamps', f'{K("created")} : STRING', f'{K("created")} : STRING , {K("updated")} : STRING',
           f'{K("updated")} : STRING')
    b.rule('Extra', f'{K("notes")} : Value', f'{K("meta")} : Object',
           f'{K("score")} : NUMBER , {K("rank")} : NUMBER',
           f'{K("owner")} : Object , {K("version")} : NUMBER')
    b.rule('Value', 'Object', 'Array', 'STRING', 'NUMBER', 'true', 'false', 'null')
    b.rule('Object', '{ }', '{ Members }')
    b.rule('Members', 'Pair', 'Members , Pair')
    b.rule('Pair', 'STRING : Value')
    b.rule('Array', '[ ]', '[ Elements ]')
    b.rule('Elements', 'Value', 'Elements , Value')
    reserved = {'"%s"' % k for k in _JSON_KEYS}
    return b.build('Root', str_chars + '"{}[]:,' + DIGIT + 'eE+-.' + 'truefalsn \n', True, reserved)


def smiles_grammar() -> GrammarSpec:
    """SMILES-like molecular-string CFG (atoms, bonds, branches in parentheses,
    ring-closure digits, bracket atoms); no whitespace terminal."""
    b = _Builder('smiles-like')
    # two-letter symbols precede their one-letter prefixes only where the
    # second letter is not itself a lexeme, so concatenation re-lexes exactly
    organic = ['Cl', 'Br', 'B', 'C', 'N', 'O', 'P', 'S', 'F', 'I']
    aromatic = ['b', 'c', 'n', 'o', 'p', 's']
    metals = ['Na', 'K', 'Fe', 'Zn', 'Mg', 'Ca', 'Li', 'Si', 'Se']
    for a in organic + aromatic + metals:
        b.lit(a)
    for c, nm in [('[', 'LB'), (']', 'RB'), ('H', 'H'), ('@@', 'AT2'), ('@', 'AT'), ('+', 'PLUS'),
                  ('-', 'MINUS'), ('=', 'EQ'), ('#', 'HASH'), ('$', 'DOLLAR'), (':', 'COLON'),
                  ('/', 'SLASH'), ('\\', 'BSLASH'), ('.', 'DOT'), ('(', 'LP'), (')', 'RP')]:
        b.lit(c, nm)
    b.term('DIGIT', '[0-9]', ('digits', 1, 1))
    b.term('PCT2', '%[0-9][0-9]', ('lit_choice', ['%10', '%11', '%12', '%23', '%42']))
    b.rule('Smiles', 'Chain')
    b.rule('Chain', 'BAtom', 'Chain BAtom', 'Chain Bond BAtom', 'Chain DOT BAtom')
    b.rule('BAtom', 'Atom', 'Atom RingBonds', 'Atom Branches', 'Atom RingBonds Branches')
    b.rule('RingBonds', 'RingBond', 'RingBonds RingBond')
    b.rule('RingBond', 'RNum', 'Bond RNum')
    b.rule('RNum', 'DIGIT', 'PCT2')
    b.rule('Branches', 'Branch', 'Branches Branch')
    b.rule('Branch', 'LP Chain RP', 'LP Bond Chain RP', 'LP DOT Chain RP')
    b.rule('Bond', 'MINUS', 'EQ', 'HASH', 'DOLLAR', 'COLON', 'Direction')
    b.rule('Direction', 'SLASH', 'BSLASH')
    b.rule('Atom', 'Organic', 'Aromatic', 'BracketAtom')
    b.rule('Organic', 'Halogen', 'Nonmetal', 'B')
    b.rule('Halogen', 'F', 'Cl', 'Br', 'I')
    b.rule('Nonmetal', 'C', 'N', 'O', 'P', 'S')
    b.rule('Aromatic', 'AromC', 'AromHetero')
    b.rule('AromC', 'c', 'b')
    b.rule('AromHetero', 'n', 'o', 'p', 's')
    b.rule('BracketAtom', 'LB BracketBody RB')
    b.rule('BracketBody', 'Isotope ElemSpec', 'ElemSpec')
    b.rule('ElemSpec', 'Symbol', 'Symbol Chiral', 'Symbol HCount', 'Symbol Charge', 'Symbol Chiral HCount',
           'Symbol HCount Charge', 'Symbol Chiral HCount Charge', 'Symbol Chiral Charge', 'Symbol Class',
           'Symbol HCount Class', 'Symbol Charge Class')
    b.rule('Isotope', 'DIGIT', 'DIGIT DIGIT', 'DIGIT DIGIT DIGIT')
    b.rule('Symbol', 'ElemSym', 'AromSym', 'Metal', 'H')
    b.rule('ElemSym', 'Halogen', 'Nonmetal', 'B')
    b.rule('AromSym', 'AromC', 'AromHetero', 'Se')
    b.rule('Metal', 'Alkali', 'Transition', 'Group2', 'Si')
    b.rule('Alkali', 'Na', 'K', 'Li')
    b.rule('Transition', 'Fe', 'Zn')
    b.rule('Group2', 'Mg', 'Ca')
    b.rule('Chiral', 'AT', 'AT2')
    b.rule('HCount', 'H', 'H DIGIT')
    b.rule('Charge', 'PosCharge', 'NegCharge')
    b.rule('PosCharge', 'PLUS', 'PLUS DIGIT', 'PLUS PLUS')
    b.rule('NegCharge', 'MINUS', 'MINUS DIGIT', 'MINUS MINUS')
    b.rule('Class', 'COLON ClassNum')
    b.rule('ClassNum', 'DIGIT', 'ClassNum DIGIT')
    charset = ''.join(sorted(set(''.join(organic + aromatic + metals) + '[]H@+-=#$:/\\.()%' + DIGIT)))
    return b.build('Smiles', charset, has_ws=False)


_OPS = ['+', '-', '*', '/', '%', '=', '==', '!=', '<', '>', '<=', '>=', '&&', '||', '!', '&', '|',
        '^', '~', '<<', '>>', '+=', '-=', '*=', '/=', '++', '--', '->', '.', ',', ';', ':', '?',
        '(', ')', '[', ']', '{', '}', '::', '#', '@', '$']
_KW_SYL = ['al', 'be', 'ca', 'de', 'el', 'fo', 'go', 'hi', 'in', 'ja', 'ke', 'lo', 'mu', 'no',
           'or', 'pe', 'qu', 're', 'st', 'tu', 'un', 'vo', 'wh', 'xe', 'yi', 'zo']


def random_grammar(seed: int, n_nt: int, n_prod: int, n_term: int, rhs_max: int,
                   rec_frac: float, left_rec: bool, name: str) -> GrammarSpec:
    """Seeded random C-like CFG.

    Terminals: keyword literals, operator literals, an identifier class, a
    number class, a string class and a skipped whitespace terminal.  Every
    nonterminal is productive and reachable (a spanning chain over the
    nonterminal order guarantees both), there are no epsilon productions
    (hence no epsilon cycles), RHS lengths are uniform in [1, rhs_max] and
    at least rec_frac of the productions are recursive (left-recursive
    ``A -> A ...`` when left_rec)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    b = _Builder(name)
    n_ops = min(len(_OPS), max(8, (n_term - 4) // 2))
    n_kw = n_term - 4 - n_ops
    kws = set()
    while len(kws) < n_kw:
        L = int(rng.integers(1, 4))
        w = ''.join(_KW_SYL[int(rng.integers(len(_KW_SYL)))] for _ in range(L))
        if len(w) <= 8:
            kws.add(w)
    kws = sorted(kws)
    for w in kws:
        b.lit(w, 'kw_' + w)
    ops = list(rng.permutation(_OPS)[:n_ops])
    for o in ops:
        b.lit(str(o), 'op_' + str(o))
    b.term('IDENT', '[a-z_][a-z0-9_]*', ('word', LOWER + '_', LOWER + DIGIT + '_', 1, 8))
    b.term('NUMBER', '[0-9]+(\\.[0-9]+)?', ('number_simple',))
    b.term('STRING', '"[a-z0-9 ]*"', ('string', LOWER + DIGIT + ' ', 0, 8))
    b.term('WS', '[ \\n]+', ('ws',), skip=True)
    T = len(b.terms)
    n_real = T - 1                                   # WS never appears in a rhs
    nts = ['N%d' % i for i in range(n_nt)]
    for nm in nts:
        b.nt(nm)
    prods = []
    # spanning chain: NT i gets a base production that mentions NT i+1 (if
    # any) and otherwise terminals; it is productive because the chain ends in
    # an all-terminal production, and every NT is reachable from N0.
    children = {i: [] for i in range(n_nt)}
    for j in range(1, n_nt):
        parent = int(rng.integers(max(0, j - 8), j))
        children[parent].append(j)

    def rand_term():
        return int(rng.integers(n_real))

    for i in range(n_nt):
        ch = children[i]
        # split children over a few base productions
        groups = [ch[k:k + 2] for k in range(0, len(ch), 2)] or [[]]
        for grp in groups:
            L = int(rng.integers(max(1, len(grp)), rhs_max + 1))
            rhs = [rand_term() for _ in range(L)]
            slots = rng.permutation(L)[:len(grp)]
            for s, c in zip(slots, grp):
                rhs[s] = T + c
            prods.append((i, rhs))
    n_rec_target = int(np.ceil(rec_frac * n_prod))
    n_rec = 0
    while len(prods) < n_prod:
        i = int(rng.integers(n_nt))
        L = int(rng.integers(1, rhs_max + 1))
        want_rec = n_rec < n_rec_target
        if want_rec and L < 2:
            L = 2
        rhs = []
        for _ in range(L):
            if rng.random() < 0.35:
                rhs.append(T + int(rng.integers(n_nt)))
            else:
                rhs.append(rand_term())
        if want_rec:
            pos = 0 if left_rec else int(rng.integers(L))
            rhs[pos] = T + i
            n_rec += 1
        prods.append((i, rhs))
    b.prods = []
    gs = GrammarSpec(name, b.terms, nts, 0, prods,
                     charset=LOWER + DIGIT + '_ "' + ''.join(sorted(set(''.join(_OPS)))),
                     has_ws=True, reserved=set(kws))
    return gs


def grammar_for(workload: str) -> GrammarSpec:
    if workload == 'expr-tiny':
        return expr_grammar()
    if workload == 'json-schema':
        return json_grammar()
    if workload == 'smiles-256':
        return smiles_grammar()
    if workload == 'clike-512':
        return random_grammar(2002, 150, 500, 100, 5, 0.15, False, 'clike-512')
    if workload == 'random-stress-1024':
        return random_grammar(3003, 400, 1500, 128, 6, 0.20, True, 'random-stress-1024')
    raise KeyError(workload)
