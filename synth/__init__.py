"""Seeded synthetic inputs (grammars, vocabularies, partial outputs,
candidates).  Shared by the tests, the benchmark and the oracle's drivers;
holds none of the validity-checking arithmetic."""
from .grammars import GrammarSpec, Terminal, grammar_for, rx_lit, rx_class  # noqa: F401
from .workload import (WORKLOADS, Workload, WorkloadSpec, make_workload,  # noqa: F401
                       sample_derivation, render, tokenize)
