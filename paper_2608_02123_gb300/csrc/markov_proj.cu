// Markov projection of one PCTree stage (Eq. 3) for float32 heads:
//
//   Z[row][v] = L_d[req(row)][v] + sum_h W_out[v][h] * X[row][h]
//
// where X[row] = E_in[parent token of row] (gathered by the previous stage),
// so that sum_h W_out[v][h] X[row][h] is the Markov head's bias for that
// parent.  A plain CUDA-core kernel with float32 accumulation (tensor cores
// would round float32 inputs to tf32); the stage logits Z go to the workspace
// and partials_kernel reduces them.  bf16 heads take markov_fused.cu, which
// never writes Z.
#include "pctree_common.cuh"

namespace pct {

namespace {

// ---------------------------------------------------------------------------
// f32 heads: CUDA-core kernel, float32 accumulation
// ---------------------------------------------------------------------------

constexpr int kF32Rows = 128;     // vocabulary rows per CTA (one per thread)
constexpr int kF32K = 32;         // K chunk staged in shared memory
constexpr int kF32Group = 8;      // parent rows per pass

__global__ void __launch_bounds__(kF32Rows)
markov_f32_kernel(const float* __restrict__ W, const float* __restrict__ X,
                  const float* __restrict__ L, long long l_req_stride,
                  float* __restrict__ Z, int ldz, int V, int H, int rows,
                  int rows_per_req, int32_t* status) {
  __shared__ float ws[kF32Rows][kF32K + 1];
  __shared__ float xs[kF32Group][kF32K];
  const int v0 = blockIdx.x * kF32Rows;
  const int v = v0 + threadIdx.x;
  bool bad = false;
  for (int g0 = 0; g0 < rows; g0 += kF32Group) {
    float acc[kF32Group];
#pragma unroll
    for (int g = 0; g < kF32Group; ++g) acc[g] = 0.0f;
    for (int h0 = 0; h0 < H; h0 += kF32K) {
      for (int i = threadIdx.x; i < kF32Rows * kF32K; i += kF32Rows) {
        const int rr = i / kF32K, hh = i % kF32K;
        const int vv = v0 + rr, h = h0 + hh;
        ws[rr][hh] = (vv < V && h < H) ? W[static_cast<size_t>(vv) * H + h] : 0.0f;
      }
      for (int i = threadIdx.x; i < kF32Group * kF32K; i += kF32Rows) {
        const int g = i / kF32K, hh = i % kF32K;
        const int row = g0 + g, h = h0 + hh;
        xs[g][hh] = (row < rows && h < H) ? X[static_cast<size_t>(row) * H + h] : 0.0f;
      }
      __syncthreads();
#pragma unroll 4
      for (int hh = 0; hh < kF32K; ++hh) {
        const float w = ws[threadIdx.x][hh];
#pragma unroll
        for (int g = 0; g < kF32Group; ++g) acc[g] = fmaf(w, xs[g][hh], acc[g]);
      }
      __syncthreads();
    }
    if (v < V) {
#pragma unroll
      for (int g = 0; g < kF32Group; ++g) {
        const int row = g0 + g;
        if (row < rows) {
          const float lval = L[static_cast<long long>(row / rows_per_req) * l_req_stride + v];
          const float z = lval + acc[g];
          bad |= isnan(z) || (isinf(z) && !(isinf(lval) && lval < 0.0f));
          Z[static_cast<size_t>(row) * ldz + v] = z;
        }
      }
    }
  }
  if (bad) set_status(status, PCTREE_ERR_NONFINITE);
}

}  // namespace

cudaError_t launch_markov_f32(const float* W_out, const float* X,
                              const float* L, long long l_req_stride, float* Z,
                              int ldz, int V, int H, int rows,
                              int rows_per_req, int32_t* status,
                              cudaStream_t stream) {
  const int grid = (V + kF32Rows - 1) / kF32Rows;
  markov_f32_kernel<<<grid, kF32Rows, 0, stream>>>(W_out, X, L, l_req_stride, Z,
                                                   ldz, V, H, rows, rows_per_req,
                                                   status);
  return cudaGetLastError();
}

}  // namespace pct
