// Kernels for float32 logits.
#define VSD_T float
#include "vsd_kernels_impl.cuh"
