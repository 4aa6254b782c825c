"""Oracle for the PVS / EAHR hot path of arXiv 2608.07152.

TEST INFRASTRUCTURE ONLY.  This package is a plain, slow, CPU implementation
of what the path computes, written from the paper and sharing no code with
the CUDA library.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import it;
the product path never does.

Modules
-------
``pvs_oracle``   PVS quantization, norm bounds, gamma_m, score intervals
                 (Sec. 2.3.1, Appendix A.1; the bound arithmetic is in
                 ``pvs_ref.c``), the one-scale quantization of the
                 scalar-quantization ablation (Sec. 3.5, 4.4), the
                 authoritative float32 score and the complete dense ranking
                 (Sec. 2.1).
``pbm_oracle``   PBM sparse scores S(x) and range bounds H(R) in the fixed
                 float32 term order (Sec. 2.3.2, Appendix A.2), block
                 maxima, and the complete sparse ranking (Sec. 2.1).
``rrf_oracle``   complete-list weighted RRF and the target T*_K (Sec. 2.1),
                 in exact rational arithmetic.
``eahr_oracle``  the ordered certification rule of Sec. 2.2 applied to given
                 ranked prefixes, used to pin stopping depths.

Parity status: every function here is pinned by a ``-m "not gpu"`` test
against a closed form, a worked case, brute force on tiny inputs or the
controlled-stream outcomes the paper reports (Sec. 4.2); none is
"parity unpinned".
"""
