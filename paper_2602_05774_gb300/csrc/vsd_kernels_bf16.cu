// Kernels for bfloat16 logits.
#define VSD_T __nv_bfloat16
#include "vsd_kernels_impl.cuh"
