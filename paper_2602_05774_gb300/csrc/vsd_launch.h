// vsd_launch.h -- host-side launchers of the VSD kernels, one set per logit
// dtype (defined in vsd_kernels_f32.cu and vsd_kernels_bf16.cu).
#pragma once

#include <cuda_runtime.h>

#include "vsd_passes.cuh"
#include "vsd_tree.cuh"

namespace vsd {

template <typename T> struct Launch {
    // z~ ~ q per row, tokens/logq/row_stats written from the row records
    static cudaError_t sample(const Problem<T>& P, bool vec, cudaStream_t s);
    // row statistics of draft+target with given tokens (linear paths)
    static cudaError_t rows_verify(const Problem<T>& P, bool vec, cudaStream_t s);
    // log kappa of supplied greedy reference paths: [B][D] rows -> out [B][D]
    static cudaError_t reference(const Problem<T>& P, bool vec, float* out, cudaStream_t s);
    // accepted lengths, residual draws, corrected paths, log-kappa (linear)
    static cudaError_t paths(const Problem<T>& P, bool vec, cudaStream_t s);
    // tree verification in one persistent launch: node rows, acceptance scan,
    // residual draws, deepest node, bonus
    static cudaError_t tree(const Problem<T>& P, bool vec, cudaStream_t s);
    // tree verification with the sequential sibling rule
    static cudaError_t tree_seq(const Problem<T>& P, bool vec, cudaStream_t s);
    // the E-step + M-step over draft trees (node rows, per-tree M-step, gradient rows)
    static cudaError_t tree_em(const Problem<T>& P, bool vec, const vsd_tree_em_outputs& o,
                               void* grad, bool grad_bf16, cudaStream_t s);
    // M-step weights and loss from an E-step view
    static cudaError_t weights(const Problem<T>& P, const EStepView& E, float* weights,
                              float* loss, cudaStream_t s);
    // gradient rows from coefficients and row statistics
    static cudaError_t grad(const Problem<T>& P, bool vec, const float4* rstats, void* grad,
                            bool grad_bf16, cudaStream_t s);
    // the fused persistent E-step + M-step kernel
    static cudaError_t fused(const Problem<T>& P, bool vec, void* grad, bool grad_bf16,
                             int ctas, cudaStream_t s);
    // resident blocks per SM of the fused kernel
    static int fused_blocks_per_sm(const Problem<T>& P, bool vec, bool grad_bf16);
};

// Host-side per-device caches, so that a call makes no attribute or
// occupancy query once a kernel has been set up on its device (vsd_api.cu).
// The SM count of the current device.
int device_sm_count();
// Lets `kernel` use `smem` bytes of dynamic shared memory on the current
// device (cudaFuncSetAttribute only when a larger size than before is asked).
cudaError_t ensure_dyn_smem(const void* kernel, size_t smem);
// Resident blocks per SM of `kernel` with `threads` threads and `smem` bytes
// of dynamic shared memory on the current device (0 on error).
int blocks_per_sm(const void* kernel, int threads, size_t smem);

inline size_t table_smem_bytes(int nch) { return (size_t)nch * sizeof(float4); }
// Dynamic shared memory of a streaming kernel: the TMA ring (vector rows
// only) followed by the chunk table.
inline size_t stream_smem_bytes(int nch, bool vec) {
    return (vec ? sizeof(Ring) : 0) + table_smem_bytes(nch);
}

// The draft LM head on the tensor cores (vsd_lmhead.cu): logits = hidden .
// weight^T, bf16 in, fp32 accumulation, bf16 out; status collects timeouts.
bool lmhead_shape_ok(const void* hidden, const void* weight, const void* logits, int M, int N,
                     int K);
// With chunk_tab, the epilogue also writes chunk_tab[r * chunk_stride + ch].xy
// = (max, sum 2^{(x - max) chunk_c}) of row r's bf16 logits x in columns
// [1024 ch, 1024 ch + 1024): the draft half of the E-step's chunk table.
cudaError_t lmhead_gemm(const void* hidden, const void* weight, int M, int N, int K, void* logits,
                        int* status, uint64_t timeout_ns, cudaStream_t s,
                        float4* chunk_tab = nullptr, int chunk_stride = 0, float chunk_c = 0.f);
// The LM head's backward (vsd_lmhead_bwd.cu): d_hidden = G . weight and
// d_weight = G^T . hidden (fp32, either may be null), with G the gradient of
// the bf16 draft logits made on chip from the E-step's row records, M-step
// coefficients and (klr non-null) top-K terms.
// fac_scratch: lmhead_backward_fac_bytes(R) bytes of device memory, 16-byte
// aligned, for the rows' packed factors.
size_t lmhead_backward_fac_bytes(int R);
cudaError_t lmhead_backward(const void* hidden, const void* weight, const void* logits, int R,
                            int V, int H, float T, const RowRec* rows, const Coef* coef,
                            const KlRec* klr, void* fac_scratch, float* d_hidden,
                            float* d_weight, int* status, uint64_t timeout_ns, cudaStream_t s);

}  // namespace vsd
