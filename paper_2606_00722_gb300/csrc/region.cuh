// Validity checks by region, for grammars whose charts are large and for
// batches with many checks per sequence.  The three steps live in
// region_forward.cu, region_good.cu and region_check.cuh (instantiated by
// region_check_sm.cu and region_check_global.cu).
//
// Every check x (+) (i, t) differs from x only around position i.  So:
//  1. k_forward: one forward chart F of x per sequence (one warp each; or
//     k_forward_block, one CTA each),
//     recording its graph (edges, gap flags), where each position's segment
//     sits in it, and each entry's completed nonterminals.  If x itself is
//     not completable, no single update is (the update's completion language
//     is a subset of x's), and every check of the sequence is 0.
//  2. k_good: a backward pass over F marks the "good" items: an item
//     (p, d, o) at node j is good if its own closure -- scanning along the
//     graph after j, nested constituents completing where F records them,
//     and its completion advancing the items waiting at column o -- reaches
//     the accepting item.  Such a closure uses only the graph after j and
//     the columns at o and before, so it is the same in every check whose
//     region lies after o and before j.
//  3. k_check: per check, only the region is walked (the candidate's span,
//     merged with fixed neighbours) with lookbacks into F; from the first
//     node after the region on, an item whose origin is an F node is
//     resolved by its good mask, and only the items whose origin lies in the
//     region are carried forward over F's graph.  The check is valid iff a
//     good item is found (or the accepting item, when the region holds the
//     start or the end).
#pragma once
#include "gscols.cuh"
#include "packs.cuh"
#include "seqpack.cuh"

