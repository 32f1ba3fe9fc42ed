// One whole PCTree drafting round (Algorithm 1, stages d = 0..B-1) in a single
// persistent, cooperative launch, for rounds with at most 16 Markov rows per
// stage (batch * k <= 16, k <= 16) -- the batch-1 drafting of Sec. 5 -- with
// either child scoring (PCTree, or the Shared-Markov control of Sec. 5.3).
//
// Per stage d, every CTA (one per SM) streams an equal share of the stage's
// (W_out tile, K chunk) pairs with TMA and multiplies them on the tensor
// cores (tcgen05, bf16 -> f32 in TMEM) against the stage's parent rows
// X = E_in[parent tokens] (Eq. 3), a 16-row buffer in global memory loaded
// with one TMA box per ring slot; a tile cut by a share boundary is finished
// by one of the two CTAs that share it (see Share below).  The
// epilogue adds the shared base logits L_d and keeps, per parent row, a
// running log-sum-exp (Eq. 2) and a warp-resident top-k list -- the stage
// logits never reach HBM.  When a CTA has finished its tiles it publishes
// per-CTA partials; the last CTA to arrive (atomic ticket, no waiting) merges
// them: per-row normaliser and top-k children, joint scores s(child) = s(p) +
// log pi (Eq. 4), the pool push, the layer-wise frontier (Sec. 4.1) and the
// next stage's parent rows, then releases a flag.  Producers keep
// prefetching the next stage's W_out tiles while that merge runs and only
// hold back the parent-row loads until the flag is set.
//
// Consecutive stages walk a CTA's (tile, chunk) pairs in opposite
// directions, so a stage begins with the data the previous stage read last;
// W_out is read with an L2 evict_first policy, so that data is the most
// likely to still sit in L2.
//
// Warp roles (320 threads): warp 0 TMA producer, warp 1 TMEM allocator + MMA
// issuer, warps 2..9 epilogue in two groups of four, group h reading TMEM
// accumulator buffer h (lane quadrant = warp % 4); the eight epilogue warps
// also run the combine and the merge, one parent row per warp.
#include <cuda_runtime.h>

#include "pctree_common.cuh"
#include "sm103_ptx.cuh"

namespace pct {
namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kUmmaK = 16;
constexpr int kBN = kFusedRows;                  // MMA N (Markov rows, max)
constexpr int kMaxKF = kFusedMaxK;               // k limit of this path
constexpr int kEpiWarps = 8;
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr int kThreads = 64 + kEpiThreads;
constexpr int kABytes = kBM * kBK * 2;           // 16 KB of W_out per slot
constexpr int kBBytes = kBN * kBK * 2;           // 2 KB of parent rows
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kStages = 8;
constexpr int kTmemCols = 32;                    // two 16-column accumulators
constexpr int kG = kFusedMaxGrid / 32;           // CTA groups of 32 in a merge
constexpr float kNegInf = -INFINITY;

template <int R>
struct FusedSmem {
  uint64_t full[kStages], empty[kStages], acc_full[2], acc_empty[2], drain;
  uint32_t tmem_slot;
  int abort;
  int ticket;
  int stop;              // snapshot of abort the epilogue warps all act on
  float lv[kEpiWarps][R][kMaxKF];          // per-warp top-k lists per row
  int lt[kEpiWarps][R][kMaxKF];
  union {
    struct {                               // per-thread (max, sum-exp)
      float m[R][kEpiThreads];
      float s[R][kEpiThreads];
    } part;
    struct {                               // merge: CTAs whose best entry
      int cta[kEpiWarps][kG * 32];         // reaches the k-th best of them
    } stage;
  } u;
  unsigned long long keys[R * kMaxKF];     // new layer: (score, id) keys
  int ktok[R * kMaxKF];                    // new layer: tokens
  int ftok[R];                             // next stage's parent tokens
  int ctok[R];                             // chain tokens (Shared-Markov)
};

template <int R>
constexpr size_t smem_bytes() {
  return 1024 + static_cast<size_t>(kStages) * kStageBytes + sizeof(FusedSmem<R>);
}

__device__ __forceinline__ void epi_barrier() { named_barrier(1, kEpiThreads); }

// This CTA's share of a stage: the contiguous range [lo, hi) of the stage's
// n_tiles * n_k (tile, K chunk) pairs numbered tile-major, lo = b * W / G for
// CTA b of G.  Every CTA gets floor(W / G) or ceil(W / G) pairs, so all of
// them stream the same number of bytes per stage.  A tile cut by a range
// boundary is shared by the two CTAs beside it (the grid never exceeds the
// tile count, so a range spans at least n_k pairs and no tile is cut twice):
// the CTA that reaches it first exports its partial accumulator, the other
// adds that partial to its own and runs the epilogue of the whole tile.
struct Share {
  int lo, hi;   // pair range
  int t0, n;    // first tile, number of (whole or partial) tiles
  __device__ __forceinline__ Share(int n_tiles, int n_k) {
    const long long W = static_cast<long long>(n_tiles) * n_k;
    lo = static_cast<int>(W * blockIdx.x / gridDim.x);
    hi = static_cast<int>(W * (blockIdx.x + 1) / gridDim.x);
    t0 = lo / n_k;
    n = (hi - 1) / n_k - t0 + 1;
  }
  // Unit i (0-based) of stage d: even stages walk the units forward, odd
  // stages backward, so each stage visits (tile, chunk) pairs in the exact
  // reverse of the previous stage's order.  [c0, c1) is the chunk range.
  __device__ __forceinline__ void unit(int d, int i, int n_k, int& tile, int& c0,
                                       int& c1) const {
    tile = t0 + ((d & 1) ? n - 1 - i : i);
    c0 = max(lo - tile * n_k, 0);
    c1 = min(hi - tile * n_k, n_k);
  }
  // CTA boundary of a cut tile: b - 1 when it begins this CTA's range,
  // b when it ends it.
  __device__ __forceinline__ int boundary(int c0) const {
    return c0 > 0 ? static_cast<int>(blockIdx.x) - 1 : static_cast<int>(blockIdx.x);
  }
};

// K chunk of the kc-th step through the range [c0, c1) in stage d.
__device__ __forceinline__ int chunk_at(int d, int kc, int c0, int c1) {
  return (d & 1) ? c1 - 1 - kc : c0 + kc;
}

// --------------------------------------------------------------------------
// producer: W_out tiles (A) and parent rows (B) into the shared-memory ring
// --------------------------------------------------------------------------

template <int R>
__device__ void produce(const CUtensorMap* tmap_w, const CUtensorMap* tmap_x,
                        const FusedArgs& a, unsigned char* ring,
                        FusedSmem<R>* S, volatile int* abort_v) {
  const Share sh(a.n_tiles, a.n_k);
  const uint64_t stream_policy = l2_policy_evict_first();
  constexpr uint32_t tx = kABytes + kBBytes;
  int stage = 0;
  uint32_t phase = 0;
  int armed[kStages];
#pragma unroll
  for (int s = 0; s < kStages; ++s) armed[s] = -1;
  int pend_stage[kStages], pend_kc[kStages];
  int n_pend = 0;                 // slots waiting for this stage's parent rows
  bool ok = true;
  auto issue_rows = [&](int st, int kx) {
    tma_load_2d(ring + st * kStageBytes + kABytes, tmap_x, &S->full[st],
                kx * kBK, 0);
  };


  for (int d = 0; d < a.B && ok; ++d) {
    bool have = d == 0;   // stage 0 rows were written before the launch
    n_pend = 0;
    for (int i = 0; i < sh.n && ok; ++i) {
      int tile, c0, c1;
      sh.unit(d, i, a.n_k, tile, c0, c1);
      for (int kc = 0; kc < c1 - c0; ++kc) {
        if (!have) {
          bool rdy = poll_flag(&a.ready[d]);
          if (!rdy && n_pend == kStages) {
            // ring full of slots waiting for the parent rows
            if (!wait_flag_bounded(&a.ready[d], abort_v, a.limit_ns)) {
              ok = false;
              break;
            }
            rdy = true;
          }
          if (rdy) {
            fence_proxy_async_global();   // rows written by another CTA
            have = true;
            for (int p = 0; p < n_pend; ++p) issue_rows(pend_stage[p], pend_kc[p]);
            n_pend = 0;
          }
        }
        if (!mbar_wait_bounded(&S->empty[stage], phase ^ 1u, abort_v, a.limit_ns)) {
          ok = false;
          break;
        }
        const int kx = chunk_at(d, kc, c0, c1);
        int wx, wy;
        w_box(a.tiled, tile, kx, a.n_k, wx, wy);
        mbar_arrive_expect_tx(&S->full[stage], tx);
        tma_load_2d_hint(ring + stage * kStageBytes, tmap_w, &S->full[stage], wx, wy,
                         stream_policy);
        if (have) {
          issue_rows(stage, kx);
        } else {
          pend_stage[n_pend] = stage;
          pend_kc[n_pend] = kx;
          ++n_pend;
        }
        armed[stage] = static_cast<int>(phase);
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (ok && !have) {
      if (!wait_flag_bounded(&a.ready[d], abort_v, a.limit_ns)) {
        ok = false;
      } else {
        fence_proxy_async_global();
        for (int p = 0; p < n_pend; ++p) issue_rows(pend_stage[p], pend_kc[p]);
      }
    }
  }
  if (!ok) {
    *abort_v = 1;
    set_status(a.status, PCTREE_ERR_TIMEOUT);
    // slots armed for W_out and a parent-row box that was never issued:
    // load whatever the row buffer holds so that their barriers complete
    fence_proxy_async_global();
    for (int p = 0; p < n_pend; ++p) issue_rows(pend_stage[p], pend_kc[p]);
  }
  // every copy issued here must land before the CTA may exit
  volatile int never = 0;
  for (int s = 0; s < kStages; ++s)
    if (armed[s] >= 0)
      mbar_wait_bounded(&S->full[s], static_cast<uint32_t>(armed[s]), &never,
                        a.limit_ns);
}

// --------------------------------------------------------------------------
// MMA issuer
// --------------------------------------------------------------------------

template <int R>
__device__ void mma(const FusedArgs& a, unsigned char* ring, FusedSmem<R>* S,
                    uint32_t tmem_base, volatile int* abort_v) {
  constexpr uint32_t idesc = idesc_bf16_f32(kBM, kBN);
  const Share sh(a.n_tiles, a.n_k);
  int stage = 0;
  uint32_t phase = 0;
  int acc = 0;
  uint32_t acc_phase = 0;
  bool ok = true;
  for (int d = 0; d < a.B && ok; ++d) {
    for (int i = 0; i < sh.n && ok; ++i) {
      int tile, c0, c1;
      sh.unit(d, i, a.n_k, tile, c0, c1);
      if (!mbar_wait_bounded(&S->acc_empty[acc], acc_phase ^ 1u, abort_v, a.limit_ns)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * kBN);
      for (int kc = 0; kc < c1 - c0; ++kc) {
        if (!mbar_wait_bounded(&S->full[stage], phase, abort_v, a.limit_ns)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t a_addr = smem_u32(ring + stage * kStageBytes);
        const uint32_t b_addr = a_addr + kABytes;
#pragma unroll
        for (int kk = 0; kk < kBK / kUmmaK; ++kk) {
          tc_mma_bf16(d_tmem, desc_kmajor_sw128(a_addr + kk * kUmmaK * 2),
                      desc_kmajor_sw128(b_addr + kk * kUmmaK * 2), idesc,
                      (kc | kk) != 0 ? 1u : 0u);
        }
        tc_commit(&S->empty[stage]);
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) break;
      tc_commit(&S->acc_full[acc]);
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
  }
  if (!ok) {
    *abort_v = 1;
    set_status(a.status, PCTREE_ERR_TIMEOUT);
  }
  tc_commit(&S->drain);
  volatile int never = 0;
  mbar_wait_bounded(&S->drain, 0, &never, a.limit_ns);
}

// --------------------------------------------------------------------------
// merge of stage d by the last CTA (the eight epilogue warps)
// --------------------------------------------------------------------------

template <int R>
__device__ void merge_stage(const CUtensorMap* tmap_w, const FusedArgs& a,
                            FusedSmem<R>* S, int d) {
  const int ew = (threadIdx.x >> 5) - 2;   // 0..7
  const int lane = threadIdx.x & 31;
  const int tid = ew * 32 + lane;          // 0..255
  const int grid = gridDim.x;
  const int b_d = d == 0 ? 1 : a.k;
  const int rpq = a.shared ? 1 : b_d;      // Markov rows per request
  const int rows = a.batch * rpq;
  const int k = a.k;
  const int n_layer = b_d * k;
  const int base = level_base(d + 1, k);
  if (d > 0) (void)ld_acquire_gpu(&a.ready[d]);   // pool of earlier stages
#pragma unroll 1
  for (int c = ew; c < rows; c += kEpiWarps) {
    const int req = c / rpq, j0 = c - req * rpq;
    // PCTree: this row's children belong to frontier slot j0.  Shared-Markov:
    // the chain row's children go to every slot of the request.
    const int j_lo = a.shared ? 0 : j0, j_hi = a.shared ? b_d : j0 + 1;
    int32_t* tok = a.pool_tok + static_cast<size_t>(req) * a.P;
    int32_t* par = a.pool_par + static_cast<size_t>(req) * a.P;
    float2* sc = a.pool_s + static_cast<size_t>(req) * a.P;
    const float* cz = a.cand_z + static_cast<size_t>(c) * grid * k;
    const int32_t* ct = a.cand_t + static_cast<size_t>(c) * grid * k;
    // Loads that do not depend on one another go out together: the parent's
    // pool id, the first (best) entry of every CTA's list and the
    // normaliser partials.  Other CTAs wrote all of these during this
    // launch: L2 loads (__ldcg), as for every cross-CTA read below -- this
    // SM's L1 may still hold the same addresses from an earlier stage.
    const int pid0 = __ldcg(a.front + req * k + j_lo);
    float fz[kG];
    int ft[kG];
#pragma unroll
    for (int u = 0; u < kG; ++u) {
      const int g = u * 32 + lane;
      fz[u] = g < grid ? __ldcg(cz + static_cast<size_t>(g) * k) : kNegInf;
      ft[u] = g < grid ? __ldcg(ct + static_cast<size_t>(g) * k) : 0x7fffffff;
    }
    // log-softmax normaliser of parent row c over all CTAs' partials (Eq. 2)
    const float lse = warp_lse_from_partials<8>(
        a.part_m + static_cast<size_t>(c) * grid,
        a.part_s + static_cast<size_t>(c) * grid, grid);
    const float2 sp0 = __ldcg(sc + pid0);
    if (lse == kNegInf && lane == 0) set_status(a.status, PCTREE_ERR_NONFINITE);
    // Every CTA list is sorted best first.  Pass 1: the top-k of the CTAs'
    // first entries; its k-th value T is a lower bound of the row's k-th
    // value (k distinct CTAs hold an entry >= T).  Pass 2: only CTAs whose
    // first entry is >= T can hold further children; their lower ranks are
    // gathered into one list and loaded in warp-wide batches.
    // The list starts from each lane's best first entry (one sort); the
    // lane's other entries are offered only where they beat the k-th of
    // those, one marked entry per lane at a time.
    float bz = fz[0];
    int bt = ft[0], bu = 0;
#pragma unroll
    for (int u = 1; u < kG; ++u) {
      const bool b = cand_better(fz[u], ft[u], bz, bt);
      bz = b ? fz[u] : bz;
      bt = b ? ft[u] : bt;
      bu = b ? u : bu;
    }
    WarpList lst;
    lst.seed(bz, bt, k);
    {
      const float tz = __shfl_sync(kFull, lst.v, k - 1);
      const int tt = __shfl_sync(kFull, lst.t, k - 1);
      unsigned marks = 0;
#pragma unroll
      for (int u = 0; u < kG; ++u)
        marks |= static_cast<unsigned>((u != bu) & cand_better(fz[u], ft[u], tz, tt)) << u;
#pragma unroll 1
      while (__any_sync(kFull, marks != 0)) {
        const int sel = marks != 0 ? __ffs(marks) - 1 : -1;
        marks &= marks - 1;
        const float cv = sel >= 0 ? pick(fz, sel) : kNegInf;
        const int cti = sel >= 0 ? pick(ft, sel) : 0x7fffffff;
        lst.offer(cv, cti, k);
      }
    }
    const float T = __shfl_sync(kFull, lst.v, k - 1);
    int* qlist = S->u.stage.cta[ew];   // CTAs that reach T
    int nq = 0;
#pragma unroll
    for (int u = 0; u < kG; ++u) {
      const bool qual = u * 32 + lane < grid && fz[u] >= T && ft[u] != 0x7fffffff;
      const unsigned q = __ballot_sync(kFull, qual);
      if (qual) qlist[nq + __popc(q & ((1u << lane) - 1u))] = u * 32 + lane;
      nq += __popc(q);
    }
    __syncwarp();
    const int km1 = k - 1;
    const int n_low = nq * km1;              // ranks 1..k-1 of those CTAs
    constexpr int kJ = 4;
#pragma unroll 1
    for (int f0 = 0; f0 < n_low; f0 += 32 * kJ) {
      float v[kJ];
      int t[kJ];
#pragma unroll
      for (int j = 0; j < kJ; ++j) {
        const int f = f0 + j * 32 + lane;
        v[j] = kNegInf;
        t[j] = 0x7fffffff;
        if (f < n_low) {
          const int g = qlist[f / km1];
          const int r = 1 + f - (f / km1) * km1;
          v[j] = __ldcg(cz + static_cast<size_t>(g) * k + r);
          t[j] = __ldcg(ct + static_cast<size_t>(g) * k + r);
        }
      }
#pragma unroll
      for (int j = 0; j < kJ; ++j) {
        const bool ok = v[j] >= T && t[j] != 0x7fffffff;
        lst.offer(ok ? v[j] : kNegInf, ok ? t[j] : 0x7fffffff, k);
      }
    }
    __syncwarp();
    int t = lst.t;
    float logpi = lst.v - lse;
    if (t < 0 || t >= a.V) {
      t = 0;
      logpi = kNegInf;
    }
    for (int j = j_lo; j < j_hi; ++j) {
      const int pid = j == j_lo ? pid0 : __ldcg(a.front + req * k + j);
      const float2 sp = j == j_lo ? sp0 : __ldcg(sc + pid);
      if (lane < k) {
        const int id = base + j * k + lane;
        const float2 sn = ff_add(sp, logpi);   // Eq. 4
        tok[id] = t;
        par[id] = pid;
        sc[id] = sn;
        const int i = req * n_layer + j * k + lane;
        S->keys[i] = (static_cast<unsigned long long>(desc_key(sn.x)) << 32) |
                     static_cast<unsigned int>(id);
        S->ktok[i] = t;
      }
    }
    if (a.shared) {                        // the chain continues (Eq. 1)
      const int top = __shfl_sync(kFull, t, 0);
      if (lane == 0) S->ctok[req] = top;
    }
  }
  if (d == a.B - 1) return;
  epi_barrier();
  // frontier of each request: the k best nodes of the new layer
  const int total = a.batch * n_layer;
  for (int i = tid; i < total; i += kEpiThreads) {
    const int req = i / n_layer;
    const unsigned long long key = S->keys[i];
    int rank = 0;
    for (int jj = req * n_layer; jj < (req + 1) * n_layer; ++jj) rank += S->keys[jj] < key;
    if (rank < k) {
      a.front[req * k + rank] = static_cast<int>(key & 0xffffffffu);
      a.xtok[req * k + rank] = S->ktok[i];
      S->ftok[req * k + rank] = S->ktok[i];
    }
  }
  epi_barrier();
  // parent rows of the next stage: X[req * k + slot] = E_in[token] (PCTree)
  // or X[req] = E_in[chain token] (Shared-Markov)
  const int* row_tok = a.shared ? S->ctok : S->ftok;
  constexpr int kU = 10;
  const int per_row = a.H / 8;
  const int total_v = a.batch * (a.shared ? 1 : k) * per_row;
  const uint4* src = static_cast<const uint4*>(a.E_in);
  uint4* dst = static_cast<uint4*>(a.X);
  for (int i0 = tid; i0 < total_v; i0 += kEpiThreads * kU) {
    uint4 tmp[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int i = i0 + u * kEpiThreads;
      if (i < total_v) {
        const int row = i / per_row, off = i - row * per_row;
        tmp[u] = src[static_cast<size_t>(row_tok[row]) * per_row + off];
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int i = i0 + u * kEpiThreads;
      if (i < total_v) {
        const int row = i / per_row, off = i - row * per_row;
        dst[static_cast<size_t>(row) * per_row + off] = tmp[u];
      }
    }
  }
  fence_proxy_async_global();   // the rows are read with TMA by every CTA
  __threadfence();
  epi_barrier();
  if (tid == 0 && d + 1 != a.stall_stage) st_release_gpu(&a.ready[d + 1], 1);
}

// --------------------------------------------------------------------------
// epilogue: TMEM -> registers, online log-sum-exp and top-k per parent row
// --------------------------------------------------------------------------

template <int R>
__device__ __forceinline__ void load_acc(uint32_t taddr, float (&acc)[R]) {
  if constexpr (R == 8) {
    uint32_t r[8];
    tmem_ld_32x32b_x8(taddr, r);
    tmem_ld_wait();
#pragma unroll
    for (int c = 0; c < 8; ++c) acc[c] = __uint_as_float(r[c]);
  } else {
    uint32_t r[16];
    tmem_ld_32x32b_x16(taddr, r);
    tmem_ld_wait();
#pragma unroll
    for (int c = 0; c < 16; ++c) acc[c] = __uint_as_float(r[c]);
  }
}

template <int R>
__device__ void epilogue(const CUtensorMap* tmap_w, const FusedArgs& a,
                         FusedSmem<R>* S, uint32_t tmem_base,
                         volatile int* abort_v) {
  const int warp = threadIdx.x >> 5;
  const int ew = warp - 2;                 // 0..7
  const int grp = ew >> 2;                 // accumulator buffer of this warp
  const int quad = warp & 3;               // TMEM lanes 32*quad .. +31
  const int lane = threadIdx.x & 31;
  const int tid = ew * 32 + lane;
  const int grid = gridDim.x;
  const int k = a.k;
  const Share sh(a.n_tiles, a.n_k);
  uint32_t acc_phase = 0;
  int g_tile = 0;                          // units issued by the MMA so far
  bool bad = false;
  for (int d = 0; d < a.B; ++d) {
    const int rpq = a.shared ? 1 : (d == 0 ? 1 : k);   // rows per request
    const int rows = a.batch * rpq;
    float m[R], s[R];
    WarpList lst[R];
#pragma unroll
    for (int c = 0; c < R; ++c) {
      m[c] = kNegInf;
      s[c] = 0.0f;
      lst[c].reset();
    }
    bool ok = true;
    bool first = true;                     // first tile of this stage
    for (int i = 0; i < sh.n; ++i, ++g_tile) {
      if ((g_tile & 1) != grp) continue;
      int tile, c0, c1;
      sh.unit(d, i, a.n_k, tile, c0, c1);
      const bool cut = c1 - c0 < a.n_k;    // a tile shared with a neighbour
      // the lanes agree before the warp-collective TMEM load
      if (!__all_sync(kFull, mbar_wait_bounded(&S->acc_full[grp], acc_phase, abort_v,
                                               a.limit_ns))) {
        ok = false;
        break;
      }
      acc_phase ^= 1u;
      tc_fence_after_sync();
      float acc[R];
      load_acc<R>(tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                      static_cast<uint32_t>(grp * kBN),
                  acc);
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(&S->acc_empty[grp]);
      if (cut) {
        const int bnd = sh.boundary(c0);
        float* xp = a.xch +
                    (static_cast<size_t>(d & 1) * kFusedMaxGrid + bnd) * (kBN * kBM) +
                    quad * 32 + lane;
        int* flag = a.xflag + bnd * 4 + quad;
        if (i == 0) {
          // first unit of the walk: hand the partial sums to the neighbour,
          // which reaches this tile as its last unit
#pragma unroll
          for (int c = 0; c < R; ++c)
            if (c < rows) __stcg(xp + c * kBM, acc[c]);
          __threadfence();
          __syncwarp();
          if (lane == 0) st_release_gpu(flag, d + 1);
          continue;
        }
        // last unit of the walk: the neighbour exported its part of this
        // tile when it began the stage
        if (!__all_sync(kFull, wait_at_least_bounded(flag, d + 1, abort_v, a.limit_ns))) {
          ok = false;
          break;
        }
#pragma unroll
        for (int c = 0; c < R; ++c)
          if (c < rows) acc[c] += __ldcg(xp + c * kBM);
      }
      const int v = tile * kBM + quad * 32 + lane;
      const bool inb = v < a.V;
      const float* Lrow = a.L + static_cast<size_t>(d) * a.V + (inb ? v : 0);
      int cur_req = -1;
      float lval = 0.0f;
#pragma unroll
      for (int c = 0; c < R; ++c) {
        if (c < rows) {
          const int req = c / rpq;
          float z = kNegInf;
          int t = 0x7fffffff;
          if (inb) {
            if (req != cur_req) {   // one base-logit load per request
              cur_req = req;
              lval = __ldg(Lrow + static_cast<size_t>(req) * a.B * a.V);
            }
            z = lval + acc[c];
            t = v;
            bad |= isnan(z) || (isinf(z) && !(isinf(lval) && lval < 0.0f));
            lse_push(m[c], s[c], z);
          }
          if (first) {
            lst[c].seed(z, t, k);   // a sort instead of 32 serial inserts
          } else {
            lst[c].offer(z, t, k);
          }
        }
      }
      first = false;
    }
    if (!ok) {
      *abort_v = 1;
      set_status(a.status, PCTREE_ERR_TIMEOUT);
    }
    // The partials and candidate lists below overwrite those of stage d-1,
    // which the last CTA of that stage may still be reading.  A CTA with
    // tiles in this stage has already waited for the flag that merge
    // releases after its reads (its parent rows needed it); check it here
    // so the order holds for every CTA.
    if (d > 0 && tid == 0 && !*abort_v &&
        !wait_flag_bounded(&a.ready[d], abort_v, a.limit_ns)) {
      *abort_v = 1;
      set_status(a.status, PCTREE_ERR_TIMEOUT);
    }
    // one decision for all eight epilogue warps, which meet at named
    // barriers below: a warp that gave up waits here for the others
    epi_barrier();
    if (tid == 0) S->stop = *abort_v;
    epi_barrier();
    if (S->stop) break;
    // per-thread (max, sum-exp) and per-warp lists to shared memory
#pragma unroll
    for (int c = 0; c < R; ++c) {
      if (c < rows) {
        S->u.part.m[c][tid] = m[c];
        S->u.part.s[c][tid] = s[c];
        if (lane < k) {
          S->lv[ew][c][lane] = lst[c].v;
          S->lt[ew][c][lane] = lst[c].t;
        }
      }
    }
    epi_barrier();
    // per-CTA partials, one row per warp (rolled: runs once per stage)
#pragma unroll 1
    for (int c = ew; c < rows; c += kEpiWarps) {
      // this CTA's normaliser partial of row c: the max over its 256
      // threads first, then one exponential per thread partial
      float mv[kEpiWarps], sv[kEpiWarps];
      float mm = kNegInf;
#pragma unroll
      for (int q = 0; q < kEpiWarps; ++q) {
        mv[q] = S->u.part.m[c][q * 32 + lane];
        sv[q] = S->u.part.s[c][q * 32 + lane];
        mm = fmaxf(mm, mv[q]);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mm = fmaxf(mm, __shfl_xor_sync(kFull, mm, o));
      float ss = 0.0f;
      if (mm > kNegInf) {
#pragma unroll
        for (int q = 0; q < kEpiWarps; ++q) ss += sv[q] * expf(mv[q] - mm);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(kFull, ss, o);
      if (lane == 0) {
        a.part_m[static_cast<size_t>(c) * grid + blockIdx.x] = mm;
        a.part_s[static_cast<size_t>(c) * grid + blockIdx.x] = ss;
      }
      // the eight warp lists, 32 / k of them per warp-wide batch: the first
      // batch is sorted in one go, the others offered
      const int per = 32 / k;
      WarpList cl;
      {
        const int w = lane / k, e = lane - w * k;
        const bool has = w < per && w < kEpiWarps;
        cl.seed(has ? S->lv[w][c][e] : kNegInf, has ? S->lt[w][c][e] : 0x7fffffff, k);
      }
#pragma unroll 1
      for (int w0 = per; w0 < kEpiWarps; w0 += per) {
        const int w = w0 + lane / k, e = lane - (lane / k) * k;
        const bool has = lane < per * k && w < kEpiWarps;
        cl.offer(has ? S->lv[w][c][e] : kNegInf, has ? S->lt[w][c][e] : 0x7fffffff, k);
      }
      if (lane < k) {   // this CTA's top-k of row c, best first
        const size_t o = (static_cast<size_t>(c) * grid + blockIdx.x) * k + lane;
        a.cand_z[o] = cl.v;
        a.cand_t[o] = cl.t;
      }
    }
    __threadfence();
    epi_barrier();
    if (tid == 0) S->ticket = atomicAdd(&a.stage_cnt[d], 1);
    epi_barrier();
    if (S->ticket == grid - 1) {
      __threadfence();
      merge_stage<R>(tmap_w, a, S, d);
    }
    epi_barrier();
  }
  if (bad) set_status(a.status, PCTREE_ERR_NONFINITE);
}

template <int R>
__global__ void __launch_bounds__(kThreads, 1)
round_fused_kernel(const __grid_constant__ CUtensorMap tmap_w,
                   const __grid_constant__ CUtensorMap tmap_x,
                   const __grid_constant__ FusedArgs a) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* ring = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  FusedSmem<R>* S = reinterpret_cast<FusedSmem<R>*>(ring + kStages * kStageBytes);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&S->full[s], 1);
      mbar_init(&S->empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&S->acc_full[i], 1);
      mbar_init(&S->acc_empty[i], 4);   // the four warps of group i
    }
    mbar_init(&S->drain, 1);
    S->abort = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tmap_w);
    tma_prefetch_desc(&tmap_x);
  }
  if (warp == 1) tmem_alloc(&S->tmem_slot, kTmemCols);
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_base = S->tmem_slot;
  volatile int* abort_v = &S->abort;
  if (warp == 0) {
    if (lane == 0) produce<R>(&tmap_w, &tmap_x, a, ring, S, abort_v);
  } else if (warp == 1) {
    if (lane == 0) mma<R>(a, ring, S, tmem_base, abort_v);
  } else {
    epilogue<R>(&tmap_w, a, S, tmem_base, abort_v);
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  if (warp == 1) tmem_dealloc(tmem_base, kTmemCols);
}

template <int R>
cudaError_t launch_r(const CUtensorMap* tmap_w, const CUtensorMap* tmap_x,
                     const FusedArgs& args, int grid, cudaStream_t stream) {
  static SmemLimit limit;
  cudaError_t e = limit.ensure(reinterpret_cast<const void*>(round_fused_kernel<R>),
                               smem_bytes<R>());
  if (e != cudaSuccess) return e;
  CUtensorMap w = *tmap_w, x = *tmap_x;
  FusedArgs a = args;
  void* params[] = {&w, &x, &a};
  return cudaLaunchCooperativeKernel(reinterpret_cast<void*>(round_fused_kernel<R>),
                                     dim3(grid), dim3(kThreads), params,
                                     smem_bytes<R>(), stream);
}

}  // namespace

cudaError_t launch_round_fused(const CUtensorMap* tmap_w,
                               const CUtensorMap* tmap_x, const FusedArgs& args,
                               int grid, cudaStream_t stream) {
  if (args.batch * args.k <= 8) return launch_r<8>(tmap_w, tmap_x, args, grid, stream);
  return launch_r<16>(tmap_w, tmap_x, args, grid, stream);
}

}  // namespace pct
