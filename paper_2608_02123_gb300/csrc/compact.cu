// pctree_compact: after acceptance, move the KV rows and the target hidden
// states of the accepted path to the slots right after the verified prefix
// (Appendix A, "Tensor implementation").
//
// Work split: one thread per 16-byte column of one (layer, plane, request)
// row block, or of one request's hidden-state rows; consecutive threads take
// consecutive columns.  Each thread checks its request's path (the indices
// are loaded eight at a time with all loads in flight, so a path costs one
// or two memory round trips, not one per node), then moves its column for
// every accepted node.  The cache is compacted in place:
// accepted indices strictly increase from a[0] = 0, so a[j] >= j and slot
// T + a[j] is never one of the slots T + 1 .. T + j - 1 already written.  A
// lane therefore loads a batch of sources before it stores the batch, and
// batches go in increasing j: no source is read after it was overwritten,
// and no two lanes touch the same bytes.
//
// The step is a pure copy: bound by HBM bandwidth, it reads and writes each
// moved row once.  Leading nodes with a[j] == j (a path down the first
// children) are already in place and are not moved.
#include "pctree_common.cuh"

namespace pct {
namespace {

constexpr int kCompactThreads = 256;
constexpr int kCompactBatch = 4;      // rows in flight per thread

struct CompactArgs {
  pctree_compact_layout lay;
  const int32_t* acc;
  const int32_t* len;
  const int32_t* prefix;
  unsigned char* cache;
  const unsigned char* hid_in;
  unsigned char* hid_out;
  int32_t* status;
  int cache_units;    // layers * planes * batch * row_vecs (< 2^31)
  int total_units;    // cache_units + batch * hidden_vecs
  int row_vecs;
  int hidden_vecs;
};

// Validity of request r's path and prefix (the rule pctree_accept follows:
// root first, then strictly increasing packed indices below N).  Returns
// the accepted length L, or -1 when the request must be left untouched;
// *j0_out is the first j >= 1 with a[j] != j (the nodes before it are
// already in their slots).  The indices are read kPathBatch at a time, every
// load of a batch issued before any is used.
constexpr int kPathBatch = 4;

__device__ __forceinline__ int checked_len(const CompactArgs& a, int r, int* T_out,
                                           int* j0_out) {
  const int B = a.lay.B, N = a.lay.N;
  const int32_t* p = a.acc + static_cast<size_t>(r) * (B + 1);
  // the length, the prefix and the first batch of indices in one round trip
  // (the indices up to B are always in bounds, whatever L is)
  const int L = __ldg(a.len + r);
  const int T = __ldg(a.prefix + r);
  int x0[kPathBatch];
#pragma unroll
  for (int u = 0; u < kPathBatch; ++u) x0[u] = u <= B ? __ldg(p + u) : 0;
  *T_out = T;
  *j0_out = 1;
  if (L < 0 || L > B || T < 0 || static_cast<long long>(T) + N > a.lay.max_slots)
    return -1;
  int prev = -1;
  bool ok = true, in_place = true;
  int j0 = L + 1;
  for (int j = 0; j <= L; j += kPathBatch) {
    int x[kPathBatch];
#pragma unroll
    for (int u = 0; u < kPathBatch; ++u)
      x[u] = j == 0 ? x0[u] : (j + u <= L ? __ldg(p + j + u) : 0);
#pragma unroll
    for (int u = 0; u < kPathBatch; ++u) {
      const int jj = j + u;
      if (jj <= L) {
        ok &= jj == 0 ? x[u] == 0 : (x[u] > prev && x[u] < N);
        prev = x[u];
        if (jj >= 1 && in_place && x[u] != jj) {
          in_place = false;
          j0 = jj;
        }
      }
    }
  }
  *j0_out = j0;
  return ok ? L : -1;
}

// Moves rows j0 .. L of one 16-byte column: row j <- row p[j] of `src`.
// Loads of a batch are issued before its stores (see the in-place argument
// above).
__device__ __forceinline__ void move_column(const unsigned char* src,
                                            unsigned char* dst, long long stride,
                                            long long dst_stride,
                                            const int32_t* p, int j0, int L) {
  for (int j = j0; j <= L; j += kCompactBatch) {
    uint4 v[kCompactBatch];
#pragma unroll
    for (int b = 0; b < kCompactBatch; ++b)
      if (j + b <= L) v[b] = *reinterpret_cast<const uint4*>(src + p[j + b] * stride);
#pragma unroll
    for (int b = 0; b < kCompactBatch; ++b)
      if (j + b <= L) *reinterpret_cast<uint4*>(dst + (j + b) * dst_stride) = v[b];
  }
}

// One thread per unit: a 16-byte column of one (layer, plane, request) row
// block, or of one request's hidden-state rows.  Consecutive threads take
// consecutive columns, so a warp's loads and stores cover 512 contiguous
// bytes of a row.
__global__ void __launch_bounds__(kCompactThreads, 4)
compact_kernel(CompactArgs a) {
  const int stride = gridDim.x * blockDim.x;
  for (int u = blockIdx.x * blockDim.x + threadIdx.x; u < a.total_units; u += stride) {
    const bool in_cache = u < a.cache_units;
    int r, col, T = 0;
    long long off;                 // byte offset of the unit's row block
    if (in_cache) {
      col = u % a.row_vecs;
      int q = u / a.row_vecs;
      r = q % a.lay.batch;
      q /= a.lay.batch;
      const int plane = q % a.lay.planes;
      const int layer = q / a.lay.planes;
      off = layer * a.lay.layer_stride + plane * a.lay.plane_stride +
            r * a.lay.request_stride;
    } else {
      const int h = u - a.cache_units;
      col = h % a.hidden_vecs;
      r = h / a.hidden_vecs;
      off = 0;
    }
    int j0;
    const int L = checked_len(a, r, &T, &j0);
    if (L < 0) {
      if (a.status != nullptr && col == 0 && (!in_cache || u < a.row_vecs * a.lay.batch))
        *a.status = PCTREE_ERR_INVALID_ARG;
      continue;
    }
    const int32_t* p = a.acc + static_cast<size_t>(r) * (a.lay.B + 1);
    if (in_cache) {
      // in place after the verified prefix; nodes already in their slots
      // (a[j] == j at the head of the path, before j0) stay
      unsigned char* base = a.cache + off + T * a.lay.slot_stride + col * 16;
      move_column(base, base, a.lay.slot_stride, a.lay.slot_stride, p, j0, L);
    } else {
      const long long hb = a.lay.hidden_bytes;
      move_column(a.hid_in + static_cast<long long>(r) * a.lay.N * hb + col * 16,
                  a.hid_out + static_cast<long long>(r) * (a.lay.B + 1) * hb + col * 16,
                  hb, hb, p, 0, L);
    }
  }
}

bool aligned16(const void* p) {
  return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

}  // namespace
}  // namespace pct

extern "C" {

pctree_status pctree_compact(const pctree_compact_layout* layout,
                             const int32_t* accepted_idx,
                             const int32_t* accepted_len,
                             const int32_t* prefix_len, void* cache,
                             const void* hidden_in, void* hidden_out,
                             int32_t* status, void* stream) {
  pct::NvtxRange range("pctree_compact");
  using pct::aligned16;
  if (layout == nullptr || accepted_idx == nullptr || accepted_len == nullptr ||
      prefix_len == nullptr)
    return PCTREE_ERR_INVALID_ARG;
  const pctree_compact_layout& l = *layout;
  if (l.batch < 1 || l.B < 1 || l.N < 1 || l.layers < 0 || l.planes < 0 ||
      l.max_slots < l.N || l.hidden_bytes < 0 || (l.hidden_bytes & 15) != 0)
    return PCTREE_ERR_INVALID_ARG;
  const bool has_cache = static_cast<long long>(l.layers) * l.planes > 0;
  if (has_cache) {
    if (cache == nullptr || !aligned16(cache) || l.row_bytes < 16 ||
        (l.row_bytes & 15) != 0 || l.slot_stride < l.row_bytes ||
        (l.slot_stride & 15) != 0 || l.request_stride < 0 ||
        (l.request_stride & 15) != 0 || l.plane_stride < 0 ||
        (l.plane_stride & 15) != 0 || l.layer_stride < 0 ||
        (l.layer_stride & 15) != 0)
      return PCTREE_ERR_INVALID_ARG;
  }
  const bool has_hidden = l.hidden_bytes > 0;
  if (has_hidden) {
    if (hidden_in == nullptr || hidden_out == nullptr || !aligned16(hidden_in) ||
        !aligned16(hidden_out))
      return PCTREE_ERR_INVALID_ARG;
    const char* a0 = static_cast<const char*>(hidden_in);
    const char* a1 = a0 + static_cast<long long>(l.batch) * l.N * l.hidden_bytes;
    const char* b0 = static_cast<const char*>(hidden_out);
    const char* b1 = b0 + static_cast<long long>(l.batch) * (l.B + 1) * l.hidden_bytes;
    if (a0 < b1 && b0 < a1) return PCTREE_ERR_INVALID_ARG;   // overlap
  }
  pct::CompactArgs a;
  a.lay = l;
  a.acc = accepted_idx;
  a.len = accepted_len;
  a.prefix = prefix_len;
  a.cache = static_cast<unsigned char*>(cache);
  a.hid_in = static_cast<const unsigned char*>(hidden_in);
  a.hid_out = static_cast<unsigned char*>(hidden_out);
  a.status = status;
  a.row_vecs = has_cache ? static_cast<int>(l.row_bytes / 16) : 1;
  a.hidden_vecs = has_hidden ? static_cast<int>(l.hidden_bytes / 16) : 1;
  const long long cache_units =
      has_cache ? static_cast<long long>(l.layers) * l.planes * l.batch * (l.row_bytes / 16) : 0;
  const long long total =
      cache_units + (has_hidden ? static_cast<long long>(l.batch) * (l.hidden_bytes / 16) : 0);
  if (total == 0) return PCTREE_OK;
  if (total >= (1ll << 31) - pct::kCompactThreads * 152ll * 4) return PCTREE_ERR_UNSUPPORTED;
  a.cache_units = static_cast<int>(cache_units);
  a.total_units = static_cast<int>(total);
  // grid-stride loop over at most two waves of the four 256-thread CTAs
  // each of the 152 SMs holds (4 rows of 16 B in flight per thread, 64 KB
  // per SM); a second wave fills SMs as first-wave CTAs retire
  long long blocks = (total + pct::kCompactThreads - 1) / pct::kCompactThreads;
  if (blocks > 152 * 8) blocks = 152 * 8;
  pct::compact_kernel<<<static_cast<int>(blocks), pct::kCompactThreads, 0,
                        static_cast<cudaStream_t>(stream)>>>(a);
  return cudaGetLastError() == cudaSuccess ? PCTREE_OK : PCTREE_ERR_CUDA;
}

}  // extern "C"
