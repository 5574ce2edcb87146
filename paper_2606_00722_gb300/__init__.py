"""GB300 (sm_103a) hot path of EPIC (arXiv 2606.00722): batched validity
checking of candidate commits under a CFG, relaxed compatible subset
selection and commit, behind the C-ABI of ``include/epic.h``."""
from .epic import (Grammar, LexTable, EpicError, build, load, validate_batch,  # noqa: F401
                   validate_batch_noalloc, measure_int_peak,
                   pick_candidates, select_compatible_subset, commit, fallback_commit, decode_step, extract_witness,
                   GAP_BIT,
                   LIB_PATH, EXPORTS)
