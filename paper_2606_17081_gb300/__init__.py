"""GB300-native KV-cache-aware routing simulation (sm_103a CUDA library + binding).

`routesim` is the Python binding of the C ABI in include/routesim.h;
`workloads` draws the seeded synthetic traces; `build` compiles the library.
"""
