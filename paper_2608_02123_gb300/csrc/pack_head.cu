// pctree_pack_head: the row-major head projection W_out [V][H] (bf16) into
// the tiled layout [ceil(V/128)][ceil(H/64)][128][64] the drafting kernels
// stream with one contiguous 16 KB copy per (vocabulary tile, K chunk).
// A plain copy kernel: each thread moves 16-byte words (8 bf16), reading and
// writing each byte once; padding rows (>= V) and columns (>= H) are zeros.
#include "pctree_common.cuh"

namespace pct {
namespace {

constexpr int kTileRows = 128;
constexpr int kChunkCols = 64;
constexpr int kWordsPerRow = kChunkCols / 8;   // 16-byte words per block row

__global__ void __launch_bounds__(256)
pack_head_kernel(const uint4* __restrict__ W, uint4* __restrict__ out, int V, int H,
                 int n_k, long long n_words) {
  const int words_per_row = H / 8;   // H % 8 == 0 for bf16 heads
  for (long long o = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
       o < n_words; o += static_cast<long long>(gridDim.x) * blockDim.x) {
    // o = ((tile * n_k + chunk) * 128 + row) * 8 + word
    const int w = static_cast<int>(o % kWordsPerRow);
    const long long q = o / kWordsPerRow;
    const int r = static_cast<int>(q % kTileRows);
    const long long tc = q / kTileRows;
    const int c = static_cast<int>(tc % n_k);
    const long long t = tc / n_k;
    const long long v = t * kTileRows + r;
    const int hw = c * kWordsPerRow + w;   // source word within the row
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (v < V && hw < words_per_row) val = W[v * words_per_row + hw];
    out[o] = val;
  }
}

}  // namespace

size_t packed_head_bytes(int V, int H) {
  const size_t n_tiles = (static_cast<size_t>(V) + kTileRows - 1) / kTileRows;
  const size_t n_k = (static_cast<size_t>(H) + kChunkCols - 1) / kChunkCols;
  return n_tiles * n_k * kTileRows * kChunkCols * 2;
}

cudaError_t launch_pack_head(const void* W, void* packed, int V, int H, int num_sms,
                             cudaStream_t stream) {
  const int n_k = (H + kChunkCols - 1) / kChunkCols;
  const long long n_words = static_cast<long long>(packed_head_bytes(V, H) / 16);
  long long blocks = (n_words + 255) / 256;
  const long long cap = static_cast<long long>(num_sms) * 8;
  if (blocks > cap) blocks = cap;
  pack_head_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
      static_cast<const uint4*>(W), static_cast<uint4*>(packed), V, H, n_k, n_words);
  return cudaGetLastError();
}

}  // namespace pct
