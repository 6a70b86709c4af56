"""FGQ (arXiv 1705.01462) hot path on GB300: ternarization, DFP activation quantization and
the grouped ternary contraction, as CUDA kernels behind the C ABI of include/fgq.h.

``fgq`` is the Python binding of libfgq.so; ``synth`` holds the seeded synthetic inputs and
workload shapes; ``build`` compiles the library.
"""
