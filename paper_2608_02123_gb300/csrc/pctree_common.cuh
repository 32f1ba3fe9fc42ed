// Shared declarations of the PCTree CUDA library: workspace layout, ranking
// keys, warp-level top-k lists and the launchers each translation unit
// provides to the host API.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>
#include <mutex>
#include <nvtx3/nvToolsExt.h>

#include "pctree.h"

namespace pct {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kChunk = 8192;          // vocabulary entries per partials work item

// ---------------------------------------------------------------------------
// workspace layout (host and device agree through this struct)
// ---------------------------------------------------------------------------

struct Layout {
  int rows_max;   // batch * k: Markov rows of a full stage
  int rows_pad;   // rows of the X buffer (multiple of 16)
  int bn;         // MMA N tile (rows per projection pass)
  int ldz;        // row stride of the stage logits Z, in floats (f32 heads)
  int n_chunks;   // vocabulary chunks per row in the partials pass (f32)
  int part_slots; // partials per row the workspace holds
  int P;          // candidate pool capacity per request
  int x_elem;     // bytes per X element
  size_t off_x, off_z, off_pm, off_ps, off_pz, off_pt;
  size_t off_pool_tok, off_pool_par, off_pool_s, off_front;
  // fused-round path: cross-CTA flags, per-CTA partials, parent tokens
  size_t off_sync, sync_bytes, off_fpm, off_fps, off_fcz, off_fct, off_xtok;
  size_t off_fxch;  // fused-round path: partial accumulators of shared tiles
  // per-stage path (bf16 heads): one word per Markov row, the best k-th
  // list entry any projection CTA holds so far, tagged with the stage
  size_t off_gthr;
  size_t total;
};

// Fused round path limits: at most kFusedRows Markov rows per stage
// (batch * k), k <= kFusedMaxK, at most kFusedMaxGrid CTAs.
constexpr int kFusedRows = 16;
constexpr int kFusedMaxK = 16;
constexpr int kFusedMaxGrid = 256;
constexpr int kFusedTileRows = 128;   // vocabulary rows per W_out tile (MMA M)

struct FusedArgs {
  const float* L;        // [batch][B][V] base logits
  int V, H, B, k, batch, P, n_k, n_tiles;
  int shared;            // 1: Shared-Markov control (one chain row per request)
  int tiled;             // 1: W_out in the tiled layout (PCTREE_HEAD_TILED)
  int32_t* pool_tok;     // [batch][P]
  int32_t* pool_par;     // [batch][P]
  float2* pool_s;        // [batch][P] joint score as (hi, lo)
  int32_t* front;        // [batch][k] frontier pool ids
  int32_t* xtok;         // [batch * k] parent tokens of the next stage
  const void* E_in;      // [V][H] bf16 Markov input rows
  void* X;               // [kFusedRows][H] bf16 parent rows of the stage
  int* stage_cnt;        // [B] CTAs done with stage d
  int* ready;            // [B] parent tokens of stage d published
  float* part_m;         // [kFusedRows][grid] per-CTA max
  float* part_s;         // [kFusedRows][grid] per-CTA sum of exp
  float* cand_z;         // [kFusedRows][grid][k] per-CTA top-k logits
  int32_t* cand_t;       // [kFusedRows][grid][k] per-CTA top-k tokens
  int* xflag;            // [grid][4] stage + 1 once a shared tile's partial is out
  float* xch;            // [2][kFusedMaxGrid][kFusedRows][128] those partials
  int32_t* status;
  unsigned long long limit_ns;   // bound of every wait (1 s)
  int stall_stage;       // test hook: stage whose release is withheld, or -1
};

// Pool id of the first node of level t (t >= 1).  Level 1 has k nodes, every
// deeper level k * k (Sec. 4.1: b_0 = 1, b_d = k afterwards).
__host__ __device__ inline int level_base(int t, int k) {
  return t <= 1 ? t : 1 + k + (t - 2) * k * k;
}

__host__ __device__ inline int level_of(int id, int k) {
  if (id == 0) return 0;
  if (id <= k) return 1;
  return 2 + (id - 1 - k) / (k * k);
}

// ---------------------------------------------------------------------------
// ranking keys
// ---------------------------------------------------------------------------

// Maps a float to a uint32 whose unsigned order is the DEScending order of
// the float (-0 and +0 equal).  NaN never reaches here (rejected earlier).
__device__ __forceinline__ uint32_t desc_key(float x) {
  x = x + 0.0f;  // -0 -> +0
  uint32_t u = __float_as_uint(x);
  uint32_t asc = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ~asc;
}

// Candidate order inside one parent: larger logit first, then lower token.
// Written with bitwise operators: short-circuit forms compile to branches,
// which diverge between lanes when the comparisons differ per lane.
__device__ __forceinline__ bool cand_better(float a, int ta, float b, int tb) {
  return (a > b) | ((a == b) & (ta < tb));
}

// a[idx] for a register array of N entries (N a power of two), by a tree of
// selects on idx's bits: an indexed read would move the array to local
// memory, and one comparison per entry may compile to divergent branches.
template <int N, typename T>
__device__ __forceinline__ T pick(const T (&a)[N], int idx) {
  T lvl[N];
#pragma unroll
  for (int j = 0; j < N; ++j) lvl[j] = a[j];
#pragma unroll
  for (int w = N / 2, b = 0; w >= 1; w /= 2, ++b) {
    const bool hi = (idx >> b) & 1;
#pragma unroll
    for (int j = 0; j < w; ++j) lvl[j] = hi ? lvl[2 * j + 1] : lvl[2 * j];
  }
  return lvl[0];
}

// ---------------------------------------------------------------------------
// warp-resident sorted top-k list: lane i < k holds entry i (best first);
// other lanes hold the sentinel (-inf, INT_MAX), worse than every entry
// ---------------------------------------------------------------------------

struct WarpList {
  float v;
  int t;
  __device__ __forceinline__ void reset() {
    v = -__int_as_float(0x7f800000);
    t = 0x7fffffff;
  }
  // Inserts the warp-uniform candidate (cv, ct), dropping the k-th entry.
  __device__ __forceinline__ void insert(float cv, int ct, int k) {
    const int lane = threadIdx.x & 31;
    const bool ahead = (lane < k) & cand_better(v, t, cv, ct);
    const int pos = __popc(__ballot_sync(kFull, ahead));
    const float uv = __shfl_up_sync(kFull, v, 1);
    const int ut = __shfl_up_sync(kFull, t, 1);
    // selects, not branches (pos == k leaves every entry below k as it is)
    const bool here = lane == pos;
    const bool down = (lane > pos) & (lane < k);
    v = here ? cv : (down ? uv : v);
    t = here ? ct : (down ? ut : t);
  }
  // Starts the list from one candidate per lane (the list must be empty):
  // a warp bitonic sort puts the best first, lanes >= k take the sentinel.
  __device__ __forceinline__ void seed(float cv, int ct, int k) {
    const int lane = threadIdx.x & 31;
    v = cv;
    t = ct;
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
      for (int j = size >> 1; j > 0; j >>= 1) {
        const float ov = __shfl_xor_sync(kFull, v, j);
        const int ot = __shfl_xor_sync(kFull, t, j);
        const bool take_best = ((lane & j) == 0) == ((lane & size) == 0);
        // both orders evaluated, then selected: a lane-dependent choice
        // between two calls compiles to divergent branches
        const bool b1 = cand_better(ov, ot, v, t);
        const bool b2 = cand_better(v, t, ov, ot);
        const bool swap = (take_best & b1) | (!take_best & b2);
        v = swap ? ov : v;
        t = swap ? ot : t;
      }
    }
    if (lane >= k) reset();
  }
  // Offers one candidate per lane (lanes with nothing pass the sentinel).
  // Every candidate better than the list's k-th entry at the start of the
  // call is inserted in turn; one that an earlier insert has pushed below
  // the k-th place lands at position >= k and is dropped by insert().
  __device__ __forceinline__ void offer(float cv, int ct, int k) {
    const float tv = __shfl_sync(kFull, v, k - 1);
    const int tt = __shfl_sync(kFull, t, k - 1);
    unsigned m = __ballot_sync(kFull, cand_better(cv, ct, tv, tt));
    while (m) {
      const int src = __ffs(m) - 1;
      m &= m - 1;
      insert(__shfl_sync(kFull, cv, src), __shfl_sync(kFull, ct, src), k);
    }
  }
};

// The k best of one row's sorted candidate lists (one per projection CTA or
// vocabulary chunk, each best first; list i at cz / ct + i * k), by a
// tournament: lane l owns lists l, l + 32, ..., holding each one's head and
// next entry in registers; each of k rounds takes the warp's best head
// ((value desc, token asc), the lane breaking exact ties of padding) and
// advances that list.  Lane r ends with the r-th best entry.  For at most
// 32 * L lists.  load() issues the first loads, so that other independent
// loads can go out before run() needs them.  The lists are read through L2
// (__ldcg): another CTA of a running kernel may have written them.
template <int L>
struct ListTournament {
  float hv[L], nv[L];
  int ht[L], nt[L], pos[L];
  const float* cz;
  const int32_t* ct;
  int k;
  __device__ __forceinline__ void load(const float* cz_, const int32_t* ct_, int n_lists,
                                       int k_) {
    cz = cz_;
    ct = ct_;
    k = k_;
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int li = 0; li < L; ++li) {
      const int id = lane + 32 * li;
      const bool ok = id < n_lists;
      const size_t o = static_cast<size_t>(ok ? id : 0) * k;
      hv[li] = ok ? __ldcg(cz + o) : -INFINITY;
      ht[li] = ok ? __ldcg(ct + o) : 0x7fffffff;
      nv[li] = ok && k > 1 ? __ldcg(cz + o + 1) : -INFINITY;
      nt[li] = ok && k > 1 ? __ldcg(ct + o + 1) : 0x7fffffff;
      pos[li] = 1;                        // list index of the entry in nv
    }
  }
  __device__ __forceinline__ void run(float& out_v, int& out_t) {
    const int lane = threadIdx.x & 31;
    out_v = -INFINITY;
    out_t = 0x7fffffff;
    for (int r = 0; r < k; ++r) {
      float bv = hv[0];
      int bt = ht[0], bl = 0;
#pragma unroll
      for (int li = 1; li < L; ++li) {
        const bool b = cand_better(hv[li], ht[li], bv, bt);
        bv = b ? hv[li] : bv;
        bt = b ? ht[li] : bt;
        bl = b ? li : bl;
      }
      float wv = bv;
      int wt = bt, wl = lane;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(kFull, wv, o);
        const int ot = __shfl_xor_sync(kFull, wt, o);
        const int ol = __shfl_xor_sync(kFull, wl, o);
        const bool take = cand_better(ov, ot, wv, wt) | ((ov == wv) & (ot == wt) & (ol < wl));
        wv = take ? ov : wv;
        wt = take ? ot : wt;
        wl = take ? ol : wl;
      }
      if (lane == r) {
        out_v = wv;
        out_t = wt;
      }
      if (lane == wl) {
#pragma unroll
        for (int li = 0; li < L; ++li) {
          if (li == bl) {
            const size_t o = static_cast<size_t>(lane + 32 * li) * k;
            hv[li] = nv[li];
            ht[li] = nt[li];
            ++pos[li];
            const bool more = pos[li] < k;
            nv[li] = more ? __ldcg(cz + o + pos[li]) : -INFINITY;
            nt[li] = more ? __ldcg(ct + o + pos[li]) : 0x7fffffff;
          }
        }
      }
    }
  }
};

template <int L>
__device__ __forceinline__ void merge_sorted_lists(const float* cz, const int32_t* ct,
                                                   int n_lists, int k, float& out_v,
                                                   int& out_t) {
  ListTournament<L> tr;
  tr.load(cz, ct, n_lists, k);
  tr.run(out_v, out_t);
}

// Online (max, sum exp) pair; m = -inf means "no finite value yet".  The
// terms exp(x), x <= 0, use the fast exponential: its relative error (a few
// 1e-7) stays far below the 1e-4 tolerance on log-probabilities.
__device__ __forceinline__ void lse_push(float& m, float& s, float z) {
  // one exponential and selects (no lane-dependent branch): a new maximum
  // rescales the sum, anything else adds exp(z - m); -inf adds nothing
  const bool up = z > m;
  const float e = __expf(up ? m - z : z - m);
  s = up ? s * e + 1.0f : (z > -__int_as_float(0x7f800000) ? s + e : s);
  m = up ? z : m;
}

__device__ __forceinline__ void lse_merge(float& m, float& s, float m2,
                                          float s2) {
  const float M = fmaxf(m, m2);
  if (M == -__int_as_float(0x7f800000)) return;
  s = s * expf(m - M) + s2 * expf(m2 - M);
  m = M;
}

// Log-sum-exp normaliser of one row (Eq. 2) from n per-chunk (max, sum-exp)
// partials, in float32: a warp max, then each lane rescales and sums its
// partials, then a warp sum.  Returns -inf when no partial is finite.  Kept
// compact: it runs once per stage from a cold instruction cache.
template <int U>
__device__ __forceinline__ float warp_lse_from_partials(const float* pm,
                                                        const float* ps,
                                                        int n) {
  const int lane = threadIdx.x & 31;
  float M = -INFINITY, S = 0.0f;
  for (int c0 = 0; c0 < n; c0 += 32 * U) {
    float mv[U], sv[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int c = c0 + u * 32 + lane;
      // written by other CTAs of a running kernel: read through L2, never
      // from this SM's (non-coherent) L1
      mv[u] = c < n ? __ldcg(pm + c) : -INFINITY;
      sv[u] = c < n ? __ldcg(ps + c) : 0.0f;
    }
    float Mc = -INFINITY;
#pragma unroll
    for (int u = 0; u < U; ++u) Mc = fmaxf(Mc, mv[u]);
    float Sc = 0.0f;
    if (Mc > -INFINITY) {
#pragma unroll
      for (int u = 0; u < U; ++u) Sc += sv[u] * expf(mv[u] - Mc);
    }
    lse_merge(M, S, Mc, Sc);
  }
  float Mw = M;
#pragma unroll 1
  for (int o = 16; o > 0; o >>= 1) Mw = fmaxf(Mw, __shfl_xor_sync(kFull, Mw, o));
  float Sw = M > -INFINITY ? S * expf(M - Mw) : 0.0f;
#pragma unroll 1
  for (int o = 16; o > 0; o >>= 1) Sw += __shfl_xor_sync(kFull, Sw, o);
  return Mw == -INFINITY ? -INFINITY : Mw + logf(Sw);
}

// Joint scores are accumulated along a path as an unevaluated float pair
// (hi, lo) with hi + lo exact: each step adds a float log-probability with
// an error-free transformation (Knuth's TwoSum), so the only rounding left is
// in the log-probabilities themselves.  hi is the score rounded to float.
__device__ __forceinline__ float2 ff_add(float2 a, float b) {
  const float s = a.x + b;
  if (!isfinite(s)) return make_float2(s, 0.0f);
  const float bb = s - a.x;
  const float e = (a.x - (s - bb)) + (b - bb) + a.y;
  const float hi = s + e;
  return make_float2(hi, e - (hi - s));
}

__device__ __forceinline__ void set_status(int32_t* status, int code) {
  atomicCAS(status, 0, code);
}

// ---------------------------------------------------------------------------
// launchers (return cudaGetLastError() of the launch)
// ---------------------------------------------------------------------------

constexpr int kMaxDevices = 64;

// NVTX range over a host scope (the enqueue of a call or of one stage):
// profilers that attach to NVTX (Nsight Systems, Nsight Compute's range
// filters) attribute the kernels launched inside it to the range.  Without
// an attached tool a push/pop costs a few nanoseconds.
class NvtxRange {
 public:
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// Raises one kernel's dynamic shared-memory limit on the current device,
// once per device: the attribute belongs to the function on one device, so a
// process that drafts on several GPUs sets it on each.  Thread-safe; a call
// that fails is retried by the next launch.
class SmemLimit {
 public:
  cudaError_t ensure(const void* fn, size_t bytes) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(mu_);
    if (done_[dev]) return cudaSuccess;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(bytes));
    if (e == cudaSuccess) done_[dev] = true;
    return e;
  }

 private:
  std::mutex mu_;
  bool done_[kMaxDevices] = {};
};

// SM count of the current device and the driver's tensor-map encoder, looked
// up once per device (api.cu).
pctree_status device_facts(int* num_sms);

// bf16 tensor map of rank 1..5 with the 128-byte swizzle (innermost box
// dimension 64 elements = 128 bytes); dims innermost first, strides_bytes for
// dimensions 1..rank-1.  Requires a prior successful device_facts call.
pctree_status encode_bf16_map_nd(CUtensorMap* map, const void* base, int rank,
                                 const uint64_t* dims,
                                 const uint64_t* strides_bytes,
                                 const uint32_t* box);

// bf16 heads: the stage's projection with the log-softmax normaliser and
// top-k folded into the epilogue (markov_fused.cu).  For rows [0, rows) it
// writes one partial per (row, CTA): part_m/part_s[row * n_parts + cta] and
// part_z/part_t[(row * n_parts + cta) * k + j], n_parts =
// fused_proj_parts(V, num_sms).  `L` points at depth d of request 0.
int fused_proj_parts(int V, int num_sms);

// Coordinates of the W_out box of (vocabulary tile, K chunk) in the tensor
// map: row-major [V][H] (x = 64 kc, y = 128 tile), or the tiled layout seen
// as a [n_tiles * n_k * 128][64] matrix (x = 0, y = 128 (tile * n_k + kc)).
__device__ __forceinline__ void w_box(int tiled, int tile, int kc, int n_k,
                                      int& x, int& y) {
  x = tiled ? 0 : kc * 64;
  y = tiled ? (tile * n_k + kc) * 128 : tile * 128;
}

// Tiled-layout bytes for V x H (pack_head.cu) and the repacking launch.
size_t packed_head_bytes(int V, int H);
cudaError_t launch_pack_head(const void* W, void* packed, int V, int H, int num_sms,
                             cudaStream_t stream);

cudaError_t launch_markov_fused(const CUtensorMap* tmap_w, const CUtensorMap* tmap_x,
                                const float* L, long long l_req_stride, int V,
                                int H, int k, int rows, int rows_per_req, int bn, int tiled,
                                int num_sms, float* part_m, float* part_s,
                                float* part_z, int32_t* part_t,
                                unsigned long long* gthr, unsigned tag,
                                int32_t* status, cudaStream_t stream);

// f32 heads: Z[row][v] = L[req(row)][v] + sum_h W_out[v][h] X[row][h] for
// rows [0, rows), req(row) = row / rows_per_req; `L` points at depth d of
// request 0, requests `l_req_stride` floats apart.  partials_kernel then
// reduces Z chunk by chunk.
cudaError_t launch_markov_f32(const float* W_out, const float* X,
                              const float* L, long long l_req_stride, float* Z,
                              int ldz, int V, int H, int rows,
                              int rows_per_req, int32_t* status,
                              cudaStream_t stream);

// One drafting round's B stages in one cooperative launch (fused path).
cudaError_t launch_round_fused(const CUtensorMap* tmap_w,
                               const CUtensorMap* tmap_x, const FusedArgs& args,
                               int grid, cudaStream_t stream);

cudaError_t launch_init(const pctree_config& c, const Layout& lay,
                        const int32_t* root, const void* E_in,
                        unsigned char* ws, int32_t* status,
                        cudaStream_t stream);

cudaError_t launch_partials(const Layout& lay, int k, int V, int rows,
                            unsigned char* ws, int32_t* status,
                            cudaStream_t stream);

// Markov rows per request at stage d: its frontier (PCTree) or the single
// chain parent (Shared-Markov control).
inline int rows_per_request(const pctree_config& c, int d) {
  return c.mode == PCTREE_MODE_SHARED ? 1 : (d == 0 ? 1 : c.k);
}

// n_parts: partials per row (vocabulary chunks of the f32 path, or the
// projection's CTAs of the bf16 path).
cudaError_t launch_merge(const pctree_config& c, const Layout& lay, int d,
                         int n_parts, const void* E_in, unsigned char* ws,
                         int32_t* status, cudaStream_t stream);

cudaError_t launch_pack(const pctree_config& c, const Layout& lay,
                        unsigned char* ws, const pctree_tree& out,
                        cudaStream_t stream);

cudaError_t launch_accept(const pctree_config& c, const pctree_tree& tree,
                          const int32_t* target, int32_t* accepted_idx,
                          int32_t* accepted_len, int32_t* bonus,
                          cudaStream_t stream);

}  // namespace pct
