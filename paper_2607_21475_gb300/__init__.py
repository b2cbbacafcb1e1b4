"""GB300-native eviction-by-design (EBD) hot path: eviction with a Poisson tail
at known inclusion probabilities, and certified Hajek decode.

The compute lives in ``libebd.so`` (CUDA for sm_103a, C ABI in include/ebd.h);
``paper_2607_21475_gb300.ebd`` is its thin Python binding and ``workloads``
draws synthetic inputs.
"""
