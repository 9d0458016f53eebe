"""GB300-native SubZero+ weight path: C-ABI CUDA library plus a thin Python binding.

``binding``   -- ctypes calls of include/zo.h (zo_create, zo_refresh, zo_perturb, zo_step, ...)
``schedule``  -- caller-side buffers and the Alg. 3 call order over the binding
``workloads`` -- synthetic workload shapes and seeded input generators
``build``     -- nvcc build of libsubzero_zo.so for sm_103a

Importing ``binding`` (or ``schedule``) loads the CUDA library and fails if it
has not been built; there is no CPU implementation in this package.
"""
