"""CPU oracle of the TurboQuant search path: test infrastructure only.

Importable only from tests/, __graft_entry__.smoke() and bench.py's CPU-baseline
leg.  It shares no code with the CUDA library.
"""
from .tq_oracle import *  # noqa: F401,F403
from .tq_oracle import (Codebook, Encoded, SearchResult, codebook, rotation,  # noqa: F401
                        gaussian_matrix, splitmix64, encode, decode, pack, unpack,
                        search, exact_knn, recall_at_k, quantized_scores, row_bytes,
                        cell_moments, marginal_pdf, allowed_mask, rank_topk, Calibration, calibrate,
                        calibration32, rotate_normalize, quantize)
