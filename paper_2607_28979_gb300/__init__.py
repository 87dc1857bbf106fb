"""GB300 (sm_103a) Mixture-of-Translators KV-cache translation.

``paper_2607_28979_gb300.mot``    ctypes binding of the C ABI in ``include/mot.h``
                                  (loads ``libmot.so``; raises ImportError if it is not built)
``paper_2607_28979_gb300.build``  compiles ``libmot.so`` from ``csrc/`` for sm_103a
"""
