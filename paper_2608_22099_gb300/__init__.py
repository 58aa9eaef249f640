"""Structure-aware banded LU dispatch on one GB300 (sm_103a).

Hot path of Lujan & Edelman, "When Structure is Silent: Opportunities for
Algorithmic Dispatch in Linear Algebra" (HPEC 2025): identify the bandwidths of
a dense fp64 matrix, convert it to LAPACK band storage, and factor the band with
partial pivoting (Sec. II-A steps 1-3; Listing 2).
"""
