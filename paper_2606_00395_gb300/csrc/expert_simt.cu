// fp32 grouped expert GEMMs (exact fp32 FMA; the fp32 layer needs a 1e-4 tolerance, which
// TF32 tensor cores cannot meet).  Same tile table as the tensor-core path: block (i, j) takes
// M-tile i of the table and 128 output columns; one thread per output column loops over the
// tile's rows, so each weight row is streamed once per tile.
//   gate/up: H[r, c] = silu(X[r] . Wg_e[c]) * (X[r] . Wu_e[c])      (App. E.2, SwiGLU)
//   down:    Y[r, c] = H[r] . Wd_e[c]
#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {
namespace {

constexpr int kCols = 128;

__global__ void __launch_bounds__(kCols)
    expert_simt_kernel(int swiglu, const float* __restrict__ A, const float* __restrict__ W0,
                       const float* __restrict__ W1, const TileEntry* __restrict__ tiles,
                       const int32_t* __restrict__ num_tiles, int K, int n_out, int b_rows,
                       float* __restrict__ out, const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  // blockIdx.x < max_tiles by the grid; a dispatch that timed out leaves the table unwritten
  if (status_timed_out(status) || static_cast<int>(blockIdx.x) >= *num_tiles) return;
  const TileEntry te = tiles[blockIdx.x];
  const int c = blockIdx.y * kCols + threadIdx.x;
  if (c >= n_out) return;
  const float* w0 = W0 + (static_cast<int64_t>(te.expert) * b_rows + c) * K;
  const float* w1 = swiglu ? W1 + (static_cast<int64_t>(te.expert) * b_rows + c) * K : nullptr;
  for (int r = 0; r < te.rows; ++r) {
    const float* a = A + static_cast<int64_t>(te.a_row0 + r) * K;
    float acc0 = 0.f, acc1 = 0.f;
    if (swiglu) {
      for (int i = 0; i < K; ++i) {
        acc0 = fmaf(a[i], w0[i], acc0);
        acc1 = fmaf(a[i], w1[i], acc1);
      }
      acc0 = acc0 / (1.0f + expf(-acc0)) * acc1;
    } else {
      for (int i = 0; i < K; ++i) acc0 = fmaf(a[i], w0[i], acc0);
    }
    out[static_cast<int64_t>(te.out_row0 + r) * n_out + c] = acc0;
  }
}

}  // namespace

cudaError_t launch_expert_simt(bool swiglu, const float* A, const float* Wb0, const float* Wb1,
                               const GemmArgs& g, cudaStream_t st) {
  if (g.max_tiles <= 0) return cudaSuccess;
  dim3 grid(g.max_tiles, (g.n_out + kCols - 1) / kCols);
  return launch_pdl(expert_simt_kernel, grid, dim3(kCols), 0, st, 1, swiglu ? 1 : 0, A, Wb0, Wb1,
                    static_cast<const TileEntry*>(g.tiles), g.num_tiles, g.K, g.n_out,
                    g.b_rows_per_expert, static_cast<float*>(g.out),
                    static_cast<const int32_t*>(g.status));
}

}  // namespace pr2
