// Selection side of a PCTree drafting round on GB300:
//   init      the root of every request (Algorithm 1, initial frontier/pool)
//   partials  per vocabulary chunk of a stage-logit row: online max / sum-exp
//             (Eq. 2) and the chunk's top-k tokens
//   merge     per request: log-softmax normaliser and top-k children of each
//             parent, joint scores (Eq. 4), pool push, layer-wise frontier
//             (Sec. 4.1) and the parents' Markov input rows for the next stage
//   pack      per request: global top-N by radix select (Sec. 4.2), breadth-
//             first packing, ancestor mask, position ids and retrieve rows
//             (Appendix A "Tensor implementation")
//   accept    per request: greedy tree walk (Sec. 4.2; Appendix A)
#include <cuda_bf16.h>

#include "pctree_common.cuh"
#include "sm103_ptx.cuh"

namespace pct {

namespace {

constexpr float kNegInf = -INFINITY;
constexpr float kPosInf = INFINITY;
constexpr float kLog2e = 1.4426950408889634f;

// Copies one Markov input row E_in[token] into X[row] (bf16: 16-byte words).
__device__ void copy_row(const void* E_in, void* X, int token, int row, int H,
                         int x_elem, int tid, int nthreads) {
  if (x_elem == 2) {
    const uint4* src = reinterpret_cast<const uint4*>(
        static_cast<const __nv_bfloat16*>(E_in) + static_cast<size_t>(token) * H);
    uint4* dst = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(X) +
                                          static_cast<size_t>(row) * H);
    for (int i = tid; i < H / 8; i += nthreads) dst[i] = src[i];
  } else {
    const float* src = static_cast<const float*>(E_in) + static_cast<size_t>(token) * H;
    float* dst = static_cast<float*>(X) + static_cast<size_t>(row) * H;
    for (int i = tid; i < H; i += nthreads) dst[i] = src[i];
  }
}

// ---------------------------------------------------------------------------
// init: pool = {root}, frontier = [root], X[r] = E_in[root_r]
// ---------------------------------------------------------------------------

__global__ void init_kernel(const int32_t* __restrict__ root, const void* E_in,
                            void* X, int32_t* pool_tok, int32_t* pool_par,
                            float2* pool_s, int32_t* front, int V, int H,
                            int P, int k, int x_elem, unsigned long long* gthr,
                            int n_gthr, int32_t* status) {
  const int r = blockIdx.x;
  // the projection's shared row thresholds start the round empty (tag 0)
  for (int i = r * blockDim.x + threadIdx.x; i < n_gthr; i += gridDim.x * blockDim.x)
    gthr[i] = 0ull;
  int tok = root[r];
  if (tok < 0 || tok >= V) {
    if (threadIdx.x == 0) set_status(status, PCTREE_ERR_INVALID_ARG);
    tok = 0;  // keep every later access in bounds
  }
  if (threadIdx.x == 0) {
    pool_tok[static_cast<size_t>(r) * P] = tok;
    pool_par[static_cast<size_t>(r) * P] = -1;
    pool_s[static_cast<size_t>(r) * P] = make_float2(0.0f, 0.0f);  // s(root) = 0
    front[static_cast<size_t>(r) * k] = 0;
  }
  copy_row(E_in, X, tok, r, H, x_elem, threadIdx.x, blockDim.x);
}

// ---------------------------------------------------------------------------
// partials: one warp per (row, chunk of kChunk logits)
// ---------------------------------------------------------------------------

constexpr int kPartWarps = 8;      // warps (work items) per CTA
constexpr int kPartVec = 4;        // float4 loads per lane and step
constexpr int kPartVals = 4 * kPartVec;        // logits per lane and step
constexpr int kPartStep = 32 * kPartVals;      // logits per warp and step

// Per (row, chunk): the chunk's (max, sum of exp) and its k best logits with
// their tokens, best first (padding (-inf, INT_MAX) when the chunk holds
// fewer than k).  The warp streams the chunk in steps of 512 logits (16 per
// lane, float4 loads, all in flight before use).  Each lane keeps an online
// max / sum of exp with one rescale per step.  The warp keeps a sorted top-k
// list; each lane marks its logits that beat the list's k-th entry and the
// warp offers one marked logit per lane at a time, so a step costs as many
// offers as its busiest lane has marks (usually none or one).
__global__ void __launch_bounds__(32 * kPartWarps, 3)
partials_kernel(const float* __restrict__ Z, int ldz, int V, int k,
                int n_chunks, int rows, float* __restrict__ part_m,
                float* __restrict__ part_s, float* __restrict__ part_z,
                int32_t* __restrict__ part_t, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const int item = blockIdx.x * kPartWarps + (threadIdx.x >> 5);
  if (item >= rows * n_chunks) return;
  const int row = item / n_chunks;
  const int chunk = item - row * n_chunks;
  const int v0 = chunk * kChunk;
  const int len = min(kChunk, V - v0);
  const float* z_row = Z + static_cast<size_t>(row) * ldz + v0;
  float m = kNegInf, s = 0.0f;
  bool bad = false;
  WarpList lst;
  lst.reset();
  // value i of this lane in the step at b is logit b + (i / 4) * 128 +
  // lane * 4 + i % 4; slots past the chunk hold -inf
  auto load_step = [&](int b, float (&z)[kPartVals]) {
#pragma unroll
    for (int j = 0; j < kPartVec; ++j) {
      const int o = b + j * 128 + lane * 4;
      if (o + 3 < len) {
        const float4 q = __ldcs(reinterpret_cast<const float4*>(z_row + o));
        z[4 * j] = q.x;
        z[4 * j + 1] = q.y;
        z[4 * j + 2] = q.z;
        z[4 * j + 3] = q.w;
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e) z[4 * j + e] = o + e < len ? z_row[o + e] : kNegInf;
      }
    }
  };
  float zn[kPartVals];
  load_step(0, zn);
#pragma unroll 1
  for (int b = 0; b < len; b += kPartStep) {
    float z[kPartVals];
#pragma unroll
    for (int i = 0; i < kPartVals; ++i) z[i] = zn[i];
    if (b + kPartStep < len) load_step(b + kPartStep, zn);   // next step in flight
    // non-finite check (NaN or +inf: not below +inf) and the step maximum
    float lm = kNegInf;
    bool nf = false;
#pragma unroll
    for (int i = 0; i < kPartVals; ++i) {
      nf |= !(z[i] < kPosInf);
      lm = fmaxf(lm, z[i]);
    }
    bad |= nf;
    if (lm > m) {
      s = m == kNegInf ? 0.0f : s * ex2_approx((m - lm) * kLog2e);
      m = lm;
    }
    if (m != kNegInf) {
      // exp(z - m) = 2^(z log2 e - m log2 e): one FMA and one ex2 per logit
      const float mb = m * kLog2e;
#pragma unroll
      for (int i = 0; i < kPartVals; ++i) s += ex2_approx(fmaf(z[i], kLog2e, -mb));
    }
    const int tbase = v0 + b + lane * 4;
    unsigned skip = 0;
    if (b == 0) {
      // first step: the list starts from the 32 lanes' best logits (a sort
      // instead of serial inserts into an empty list); the lowest index
      // holding the lane's maximum has the lowest token among equal logits
      int li = 0;
#pragma unroll
      for (int i = kPartVals - 1; i >= 0; --i)
        if (z[i] == lm) li = i;
      const int lt = lm > kNegInf ? tbase + (li >> 2) * 128 + (li & 3) : 0x7fffffff;
      lst.seed(lm > kNegInf ? lm : kNegInf, lt, k);
      if (lm > kNegInf) skip = 1u << li;
    }
    // logits that beat the list's k-th entry (out-of-range slots hold -inf
    // and the sentinel token, which beats nothing); a lane whose maximum is
    // below the k-th value holds none, and most steps have no such lane
    const float tv = __shfl_sync(kFull, lst.v, k - 1);
    const int tt = __shfl_sync(kFull, lst.t, k - 1);
    if (!__any_sync(kFull, lm >= tv)) continue;
    unsigned marks = 0;
#pragma unroll
    for (int i = 0; i < kPartVals; ++i) {
      const int o = b + (i >> 2) * 128 + lane * 4 + (i & 3);
      const int tok = o < len ? tbase + (i >> 2) * 128 + (i & 3) : 0x7fffffff;
      marks |= static_cast<unsigned>(cand_better(z[i], tok, tv, tt)) << i;
    }
    marks &= ~skip;
    while (__any_sync(kFull, marks != 0)) {
      const int sel = marks != 0 ? __ffs(marks) - 1 : -1;
      marks &= marks - 1;
      const float cv = sel >= 0 ? pick(z, sel) : kNegInf;
      const int ct = sel >= 0 ? tbase + (sel >> 2) * 128 + (sel & 3) : 0x7fffffff;
      lst.offer(cv, ct, k);
    }
  }
  if (bad) set_status(status, PCTREE_ERR_NONFINITE);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(kFull, m, o);
    const float s2 = __shfl_xor_sync(kFull, s, o);
    lse_merge(m, s, m2, s2);
  }
  const size_t p = static_cast<size_t>(row) * n_chunks + chunk;
  if (lane == 0) {
    part_m[p] = m;
    part_s[p] = s;
  }
  if (lane < k) {
    part_z[p * k + lane] = lst.v;
    part_t[p * k + lane] = lst.t;
  }
}

// ---------------------------------------------------------------------------
// merge: one CTA per request, one warp per parent slot
// ---------------------------------------------------------------------------

constexpr int kUnroll = 8;

// Copies the Markov input rows of the next stage, X[first_row + slot] =
// E_in[tok[slot]] for slot < n_rows, with all loads of a batch in flight.
__device__ void gather_rows(const void* E_in, void* X, const int* tok,
                            int n_rows, int first_row, int H, int x_elem) {
  const int tid = threadIdx.x, nt = blockDim.x;
  if (x_elem == 2) {
    const int per_row = H / 8;
    const int total = n_rows * per_row;
    const uint4* src = static_cast<const uint4*>(E_in);
    uint4* dst = static_cast<uint4*>(X);
    for (int i0 = tid; i0 < total; i0 += nt * 4) {
      uint4 tmp[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * nt;
        if (i < total) {
          const int slot = i / per_row, off = i - slot * per_row;
          tmp[u] = src[static_cast<size_t>(tok[slot]) * per_row + off];
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * nt;
        if (i < total) {
          const int slot = i / per_row, off = i - slot * per_row;
          dst[static_cast<size_t>(first_row + slot) * per_row + off] = tmp[u];
        }
      }
    }
  } else {
    const int total = n_rows * H;
    const float* src = static_cast<const float*>(E_in);
    float* dst = static_cast<float*>(X);
    for (int i = tid; i < total; i += nt) {
      const int slot = i / H, off = i - slot * H;
      dst[static_cast<size_t>(first_row + slot) * H + off] =
          src[static_cast<size_t>(tok[slot]) * H + off];
    }
  }
}

// The k best of a row's candidate lists (n_cand entries, list after list)
// for any number of lists, where merge_sorted_lists would need more than 5
// lists per lane: every lane offers its candidates that beat the warp list's
// k-th entry, after a seed from each lane's best of the first batch.
__device__ __forceinline__ void merge_lists_scan(const float* __restrict__ cz,
                                                 const int32_t* __restrict__ ct,
                                                 int n_cand, int k, float& out_v,
                                                 int& out_t) {
  const int lane = threadIdx.x & 31;
  WarpList lst;
  lst.reset();
  for (int c0 = 0; c0 < n_cand; c0 += 32 * kUnroll) {
    float cv[kUnroll];
    int ci[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int c = c0 + u * 32 + lane;
      cv[u] = c < n_cand ? cz[c] : kNegInf;
      ci[u] = c < n_cand ? ct[c] : 0x7fffffff;
    }
    unsigned skip = 0;
    if (c0 == 0) {
      float bv = cv[0];
      int bi = ci[0], bu = 0;
#pragma unroll
      for (int u = 1; u < kUnroll; ++u) {
        const bool b = cand_better(cv[u], ci[u], bv, bi);
        bv = b ? cv[u] : bv;
        bi = b ? ci[u] : bi;
        bu = b ? u : bu;
      }
      lst.seed(bv, bi, k);
      skip = 1u << bu;
    }
    const float tv = __shfl_sync(kFull, lst.v, k - 1);
    const int tt = __shfl_sync(kFull, lst.t, k - 1);
    unsigned marks = 0;
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      marks |= static_cast<unsigned>(cand_better(cv[u], ci[u], tv, tt)) << u;
    marks &= ~skip;
    while (__any_sync(kFull, marks != 0)) {
      const int sel = marks != 0 ? __ffs(marks) - 1 : -1;
      marks &= marks - 1;
      const float ov = sel >= 0 ? pick(cv, sel) : kNegInf;
      const int ot = sel >= 0 ? pick(ci, sel) : 0x7fffffff;
      lst.offer(ov, ot, k);
    }
  }
  out_v = lst.v;
  out_t = lst.t;
}

constexpr int kMergeThreads = 1024;

__global__ void __launch_bounds__(kMergeThreads)
merge_kernel(int d, int B, int k, int b_d, int rpq, int shared, int V, int H,
             int P, int n_chunks,
             int x_elem, const float* __restrict__ part_m,
             const float* __restrict__ part_s,
             const float* __restrict__ part_z,
             const int32_t* __restrict__ part_t, int32_t* pool_tok,
             int32_t* pool_par, float2* pool_s, int32_t* front,
             const void* E_in, void* X, int32_t* status) {
  const int r = blockIdx.x;
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  // launched while the stage's projection finishes: wait for it before
  // reading its partials; the next stage's projection may launch meanwhile
  pdl_launch_dependents();
  pdl_wait();
  // the layer's b_d * k (score, id) keys, then their tokens
  extern __shared__ unsigned long long sm_keys[];
  int* sm_ctok = reinterpret_cast<int*>(sm_keys + b_d * k);
  __shared__ float sm_lse[32];
  __shared__ int sm_tok[PCTREE_MAX_K];
  __shared__ int sm_chain;

  int32_t* tok = pool_tok + static_cast<size_t>(r) * P;
  int32_t* par = pool_par + static_cast<size_t>(r) * P;
  float2* sc = pool_s + static_cast<size_t>(r) * P;
  int32_t* fr = front + static_cast<size_t>(r) * k;
  const int base = level_base(d + 1, k);

  // Warp j < rpq takes Markov row j of the request (a frontier slot, or the
  // chain parent of the Shared-Markov control, rpq = 1): its children; warp
  // rpq + j, when there is one, meanwhile the row's normaliser.
  const int n_warps = kMergeThreads / 32;
  const bool lse_apart = 2 * rpq <= n_warps;
  if (lse_apart && warp >= rpq && warp < 2 * rpq) {
    const size_t p0 = static_cast<size_t>(r * rpq + warp - rpq) * n_chunks;
    // log-softmax normaliser from the chunk partials (Eq. 2)
    const float lse = warp_lse_from_partials<kUnroll>(part_m + p0, part_s + p0, n_chunks);
    if (lane == 0) sm_lse[warp - rpq] = lse;
  }
  float cv = kNegInf;
  int cv_t = 0x7fffffff;
  const int j = warp;
  // the parent of slot j and its score, loaded before they are needed
  int pid = 0;
  float2 spid = make_float2(0.0f, 0.0f);
  if (j < rpq && !shared) {
    pid = fr[j];
    spid = sc[pid];
  }
  if (j < rpq) {
    const size_t p0 = static_cast<size_t>(r * rpq + j) * n_chunks;
    if (!lse_apart) {
      const float lse = warp_lse_from_partials<kUnroll>(part_m + p0, part_s + p0, n_chunks);
      if (lane == 0) sm_lse[j] = lse;
    }
    // top-k children of this parent over every chunk's list (a tournament
    // for up to 160 lists, which fits the register budget of a 1024-thread
    // block; more lists take the scan)
    const float* cz = part_z + p0 * k;
    const int32_t* ct = part_t + p0 * k;
    switch ((n_chunks + 31) / 32) {
      case 1: merge_sorted_lists<1>(cz, ct, n_chunks, k, cv, cv_t); break;
      case 2: merge_sorted_lists<2>(cz, ct, n_chunks, k, cv, cv_t); break;
      case 3: merge_sorted_lists<3>(cz, ct, n_chunks, k, cv, cv_t); break;
      case 4: merge_sorted_lists<4>(cz, ct, n_chunks, k, cv, cv_t); break;
      case 5: merge_sorted_lists<5>(cz, ct, n_chunks, k, cv, cv_t); break;
      default: merge_lists_scan(cz, ct, n_chunks * k, k, cv, cv_t); break;
    }
  }
  __syncthreads();
  if (j < rpq) {
    const float lse = sm_lse[j];
    if (lse == kNegInf && lane == 0) set_status(status, PCTREE_ERR_NONFINITE);
    int t = cv_t;
    float logpi = cv - lse;
    if (t < 0 || t >= V) {  // only when V < k (rejected on the host)
      t = 0;
      logpi = kNegInf;
    }
    // PCTree: the row's children belong to slot j; Shared-Markov: the chain
    // row's children go to every slot of the request.
    // The layer's keys and tokens also go to shared memory for the
    // frontier below.
    const int j_lo = shared ? 0 : j, j_hi = shared ? b_d : j + 1;
    for (int jj = j_lo; jj < j_hi; ++jj) {
      const int p = shared ? fr[jj] : pid;
      const float2 sp = shared ? sc[p] : spid;
      if (lane < k) {
        const int id = base + jj * k + lane;
        const float2 s_id = ff_add(sp, logpi);  // Eq. 4: s(child) = s(p) + log pi
        tok[id] = t;
        par[id] = p;
        sc[id] = s_id;
        sm_keys[jj * k + lane] =
            (static_cast<unsigned long long>(desc_key(s_id.x)) << 32) |
            static_cast<unsigned int>(id);
        sm_ctok[jj * k + lane] = t;
      }
    }
    const int top = __shfl_sync(kFull, t, 0);
    if (lane == 0 && j == 0) sm_chain = top;   // argmax of the row (Eq. 1)
  }
  if (d == B - 1) return;
  __syncthreads();
  // frontier: the k best nodes of this layer by (score desc, id asc)
  const int n_layer = b_d * k;
  for (int i = threadIdx.x; i < n_layer; i += blockDim.x) {
    const unsigned long long key = sm_keys[i];
    int rank = 0;
    for (int j = 0; j < n_layer; ++j) rank += sm_keys[j] < key;
    if (rank < k) {
      fr[rank] = base + i;
      sm_tok[rank] = sm_ctok[i];
    }
  }
  __syncthreads();
  // Markov input rows of the next stage: X[r * k + slot] = E_in[token]
  // (PCTree) or X[r] = E_in[chain token] (Shared-Markov)
  if (shared) {
    if (threadIdx.x == 0) sm_tok[0] = sm_chain;
    __syncthreads();
    gather_rows(E_in, X, sm_tok, 1, r, H, x_elem);
  } else {
    gather_rows(E_in, X, sm_tok, k, r * k, H, x_elem);
  }
}

// ---------------------------------------------------------------------------
// pack: one CTA of 1024 threads per request
// ---------------------------------------------------------------------------

constexpr int kPackThreads = 1024;

__device__ __forceinline__ int block_excl_scan(int x, int* sm_warp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = x;
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) sm_warp[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    int w = lane < nw ? sm_warp[lane] : 0;
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, w, o);
      if (lane >= o) w += y;
    }
    if (lane < nw) sm_warp[lane] = w;  // inclusive per warp
  }
  __syncthreads();
  const int before = (warp == 0 ? 0 : sm_warp[warp - 1]) + incl - x;
  if (total) *total = sm_warp[(blockDim.x >> 5) - 1];
  __syncthreads();
  return before;
}

__global__ void __launch_bounds__(kPackThreads)
pack_kernel(int B, int k, int N, int P, int pos_offset,
            const int32_t* __restrict__ pool_tok,
            const int32_t* __restrict__ pool_par,
            const float2* __restrict__ pool_s, pctree_tree out) {
  const int r = blockIdx.x;
  const int tid = threadIdx.x;
  extern __shared__ unsigned long long sm_key[];  // P keys; later reused
  __shared__ unsigned int sm_hist[256];
  __shared__ int sm_warp[32];
  __shared__ int sm_sel[PCTREE_MAX_N];    // packed index -> pool id
  __shared__ int sm_par[PCTREE_MAX_N];    // packed index -> packed parent
  __shared__ unsigned char sm_haschild[PCTREE_MAX_N];
  __shared__ unsigned long long sm_prefix;
  __shared__ int sm_remaining, sm_count;

  const int32_t* tok = pool_tok + static_cast<size_t>(r) * P;
  const int32_t* par = pool_par + static_cast<size_t>(r) * P;
  const float2* sc = pool_s + static_cast<size_t>(r) * P;
  const int n = min(N, P);

  // 46-bit keys: descending fp32 score in bits 45..14, pool id in 13..0.
  // Ids grow with depth, so (score desc, id asc) is (score desc, depth asc,
  // id asc) of Sec. 4.2.
  for (int i = tid; i < P; i += blockDim.x) {
    sm_key[i] = (static_cast<unsigned long long>(desc_key(sc[i].x)) << 14) |
                static_cast<unsigned long long>(i);
  }
  if (tid == 0) {
    sm_prefix = 0ull;
    sm_remaining = n;
  }
  __syncthreads();
  // radix select of the n-th smallest key, 8 bits per pass from bit 40
  unsigned long long mask = 0ull;
  for (int shift = 40; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += blockDim.x) sm_hist[i] = 0u;
    __syncthreads();
    const unsigned long long prefix = sm_prefix;
    for (int i = tid; i < P; i += blockDim.x) {
      const unsigned long long key = sm_key[i];
      if ((key & mask) == prefix) atomicAdd(&sm_hist[(key >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (tid < 32) {
      // lane L owns bins 8L .. 8L+7
      int cnt = 0;
      for (int b = 0; b < 8; ++b) cnt += sm_hist[tid * 8 + b];
      int incl = cnt;
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFull, incl, o);
        if (tid >= o) incl += y;
      }
      const int need = sm_remaining;
      const int excl = incl - cnt;
      const bool here = excl < need && incl >= need;
      if (here) {
        int acc = excl;
        for (int b = 0; b < 8; ++b) {
          const int hb = sm_hist[tid * 8 + b];
          if (acc + hb >= need) {
            sm_prefix = prefix | (static_cast<unsigned long long>(tid * 8 + b) << shift);
            sm_remaining = need - acc;
            break;
          }
          acc += hb;
        }
      }
    }
    mask |= 255ull << shift;
    __syncthreads();
  }
  const unsigned long long kth = sm_prefix;  // n-th smallest key, exactly
  // gather the selected pool ids (unordered) into sm_sel
  if (tid == 0) sm_count = 0;
  __syncthreads();
  for (int i = tid; i < P; i += blockDim.x) {
    if (sm_key[i] <= kth) sm_sel[atomicAdd(&sm_count, 1)] = i;
  }
  __syncthreads();
  // breadth-first packing: level by level, (parent's index, token) order
  int* pidx = reinterpret_cast<int*>(sm_key);  // pool id -> packed index
  for (int i = tid; i < P; i += blockDim.x) pidx[i] = -1;
  const int my_id = tid < n ? sm_sel[tid] : -1;
  const int my_lvl = my_id >= 0 ? level_of(my_id, k) : -1;
  // parent and token of this thread's node, loaded once: the level loop
  // below touches shared memory only
  const int my_pid = my_id >= 0 ? par[my_id] : -1;
  const int my_tok = my_id >= 0 ? tok[my_id] : 0;
  __shared__ unsigned long long sm_k2[PCTREE_MAX_N];
  __shared__ int sm_kid[PCTREE_MAX_N];
  __shared__ int sm_lvl_cnt[2];   // nodes of the current level, by parity
  if (tid == 0) sm_lvl_cnt[0] = 0;
  __syncthreads();
  int placed = 0;
  for (int t = 0; t <= B; ++t) {
    // the level's nodes take slots; the counter of the next level (last
    // read before the previous barrier) is cleared meanwhile
    const bool at = my_lvl == t;
    unsigned long long key2 = 0ull;
    if (at) {
      const int pp = (t == 0 || my_pid < 0 || my_pid >= P) ? -1 : pidx[my_pid];
      key2 = (static_cast<unsigned long long>(static_cast<unsigned int>(pp + 1)) << 32) |
             static_cast<unsigned int>(my_tok);
      const int slot = atomicAdd(&sm_lvl_cnt[t & 1], 1);
      sm_k2[slot] = key2;
      sm_kid[slot] = my_id;
    }
    if (tid == 0) sm_lvl_cnt[(t + 1) & 1] = 0;
    __syncthreads();
    const int n_t = sm_lvl_cnt[t & 1];
    if (n_t == 0) break;   // the selection is ancestor-closed: no deeper level
    // rank among the nodes of this level (<= n of them).  Siblings carry
    // distinct tokens, so (parent, token) is unique; the pool id breaks ties
    // anyway so that every packed slot is written exactly once whatever the
    // pool holds (e.g. after a round already flagged non-finite).
    if (at) {
      int rank = 0;
      for (int j = 0; j < n_t; ++j)
        rank += sm_k2[j] < key2 || (sm_k2[j] == key2 && sm_kid[j] < my_id);
      const int a = placed + rank;
      pidx[my_id] = a;
      sm_sel[a] = my_id;  // safe: sm_sel is not read inside this loop
    }
    placed += n_t;
    __syncthreads();
  }
  // per packed node: parent index, child flags
  // A parent is packed before its children (ids grow with depth and the
  // selection is ancestor-closed), so sm_par[a] < a; anything else is
  // recorded as "no parent", which keeps every walk below finite.
  for (int a = tid; a < n; a += blockDim.x) {
    const int id = sm_sel[a];
    const int pid = par[id];
    int pa = (a == 0 || pid < 0 || pid >= P) ? -1 : pidx[pid];
    if (pa >= a) pa = -1;
    sm_par[a] = pa;
    sm_haschild[a] = 0;
  }
  __syncthreads();
  for (int a = tid; a < n; a += blockDim.x)
    if (sm_par[a] >= 0) sm_haschild[sm_par[a]] = 1;
  __syncthreads();
  int32_t* o_tok = out.tokens + static_cast<size_t>(r) * N;
  int32_t* o_par = out.parent + static_cast<size_t>(r) * N;
  int32_t* o_dep = out.depth + static_cast<size_t>(r) * N;
  float* o_lp = out.logp + static_cast<size_t>(r) * N;
  int32_t* o_pos = out.position_ids + static_cast<size_t>(r) * N;
  uint8_t* o_mask = out.mask + static_cast<size_t>(r) * N * N;
  int32_t* o_ret = out.retrieve + static_cast<size_t>(r) * N * (B + 1);
  for (int a = tid; a < N; a += blockDim.x) {
    if (a < n) {
      const int id = sm_sel[a];
      const int lvl = level_of(id, k);
      o_tok[a] = tok[id];
      o_par[a] = sm_par[a];
      o_dep[a] = lvl;
      o_lp[a] = sc[id].x;
      o_pos[a] = lvl + pos_offset;  // siblings share a position (Appendix A)
    } else {
      o_tok[a] = -1;
      o_par[a] = -1;
      o_dep[a] = -1;
      o_lp[a] = kNegInf;
      o_pos[a] = -1;
    }
  }
  // leaves in packed order
  const int is_leaf = (tid < n && !sm_haschild[tid]) ? 1 : 0;
  int n_leaves;
  const int leaf_rank = block_excl_scan(is_leaf, sm_warp, &n_leaves);
  // clear mask and retrieve, then scatter the ancestor chains
  const size_t mask_bytes = static_cast<size_t>(N) * N;
  for (size_t i = tid; i < mask_bytes; i += blockDim.x) o_mask[i] = 0;
  const int ret_len = N * (B + 1);
  for (int i = tid; i < ret_len; i += blockDim.x) o_ret[i] = -1;
  __syncthreads();
  if (tid < n) {
    // ancestor-or-self mask row (the prefix is visible to every node)
    for (int b = tid; b >= 0; b = sm_par[b]) o_mask[static_cast<size_t>(tid) * N + b] = 1;
    if (is_leaf) {
      int32_t* row = o_ret + static_cast<size_t>(leaf_rank) * (B + 1);
      int dpt = level_of(sm_sel[tid], k);
      for (int b = tid; b >= 0 && dpt >= 0; b = sm_par[b]) row[dpt--] = b;
    }
  }
  if (tid == 0) {
    out.n_nodes[r] = n;
    out.n_leaves[r] = n_leaves;
  }
  if (out.pool_token != nullptr) {
    for (int i = tid; i < P; i += blockDim.x) {
      out.pool_token[static_cast<size_t>(r) * P + i] = tok[i];
      out.pool_parent[static_cast<size_t>(r) * P + i] = par[i];
      out.pool_logp[static_cast<size_t>(r) * P + i] = sc[i].x;
    }
  }
}

// ---------------------------------------------------------------------------
// accept: one warp per request
// ---------------------------------------------------------------------------

__global__ void accept_kernel(int B, int N, const int32_t* __restrict__ n_nodes,
                              const int32_t* __restrict__ tokens,
                              const int32_t* __restrict__ parent,
                              const int32_t* __restrict__ target,
                              int32_t* accepted_idx, int32_t* accepted_len,
                              int32_t* bonus, int batch) {
  const int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (r >= batch) return;
  const int lane = threadIdx.x & 31;
  // a caller-built tree may claim more nodes than its rows hold: walk at most
  // the N rows of the request
  const int n = min(max(n_nodes[r], 0), N);
  const int32_t* tk = tokens + static_cast<size_t>(r) * N;
  const int32_t* pa = parent + static_cast<size_t>(r) * N;
  const int32_t* tg = target + static_cast<size_t>(r) * N;
  int32_t* acc = accepted_idx + static_cast<size_t>(r) * (B + 1);
  for (int i = lane; i <= B; i += 32) acc[i] = -1;
  __syncwarp();
  int cur = 0, len = 0;
  if (lane == 0) acc[0] = 0;
  while (len < B) {
    const int want = tg[cur];
    int next = -1;
    // children of `cur` have indices > cur; siblings carry distinct tokens
    for (int c0 = cur + 1; c0 < n && next < 0; c0 += 32) {
      const int c = c0 + lane;
      const bool hit = c < n && pa[c] == cur && tk[c] == want;
      const unsigned m = __ballot_sync(kFull, hit);
      if (m) next = c0 + __ffs(m) - 1;
    }
    if (next < 0) break;
    cur = next;
    ++len;
    if (lane == 0) acc[len] = cur;
  }
  if (lane == 0) {
    accepted_len[r] = len;
    bonus[r] = tg[cur];
  }
}

}  // namespace

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------

cudaError_t launch_init(const pctree_config& c, const Layout& lay,
                        const int32_t* root, const void* E_in,
                        unsigned char* ws, int32_t* status,
                        cudaStream_t stream) {
  init_kernel<<<c.batch, 256, 0, stream>>>(
      root, E_in, ws + lay.off_x, reinterpret_cast<int32_t*>(ws + lay.off_pool_tok),
      reinterpret_cast<int32_t*>(ws + lay.off_pool_par),
      reinterpret_cast<float2*>(ws + lay.off_pool_s),
      reinterpret_cast<int32_t*>(ws + lay.off_front), c.V, c.H, lay.P, c.k,
      lay.x_elem, reinterpret_cast<unsigned long long*>(ws + lay.off_gthr),
      lay.rows_max, status);
  return cudaGetLastError();
}

cudaError_t launch_partials(const Layout& lay, int k, int V, int rows,
                            unsigned char* ws, int32_t* status,
                            cudaStream_t stream) {
  const int items = rows * lay.n_chunks;
  const int grid = (items + kPartWarps - 1) / kPartWarps;
  partials_kernel<<<grid, 32 * kPartWarps, 0, stream>>>(
      reinterpret_cast<const float*>(ws + lay.off_z), lay.ldz, V, k,
      lay.n_chunks, rows, reinterpret_cast<float*>(ws + lay.off_pm),
      reinterpret_cast<float*>(ws + lay.off_ps),
      reinterpret_cast<float*>(ws + lay.off_pz),
      reinterpret_cast<int32_t*>(ws + lay.off_pt), status);
  return cudaGetLastError();
}

cudaError_t launch_merge(const pctree_config& c, const Layout& lay, int d,
                         int n_parts, const void* E_in, unsigned char* ws,
                         int32_t* status, cudaStream_t stream) {
  const int b_d = d == 0 ? 1 : c.k;
  const int rpq = rows_per_request(c, d);
  const size_t smem =
      static_cast<size_t>(b_d) * c.k * (sizeof(unsigned long long) + sizeof(int));
  // 1024 threads: the normalisers beside the children, and the next stage's
  // rows gathered with every load of a row in flight.  Programmatic
  // dependent launch: scheduled while the projection finishes (the kernel
  // waits for it before touching memory).
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(c.batch);
  cfg.blockDim = dim3(kMergeThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(
      &cfg, merge_kernel,
      d, c.B, c.k, b_d, rpq, c.mode == PCTREE_MODE_SHARED ? 1 : 0, c.V, c.H,
      lay.P, n_parts, lay.x_elem,
      reinterpret_cast<const float*>(ws + lay.off_pm),
      reinterpret_cast<const float*>(ws + lay.off_ps),
      reinterpret_cast<const float*>(ws + lay.off_pz),
      reinterpret_cast<const int32_t*>(ws + lay.off_pt),
      reinterpret_cast<int32_t*>(ws + lay.off_pool_tok),
      reinterpret_cast<int32_t*>(ws + lay.off_pool_par),
      reinterpret_cast<float2*>(ws + lay.off_pool_s),
      reinterpret_cast<int32_t*>(ws + lay.off_front), E_in, ws + lay.off_x,
      status);
}

cudaError_t launch_pack(const pctree_config& c, const Layout& lay,
                        unsigned char* ws, const pctree_tree& out,
                        cudaStream_t stream) {
  const size_t smem = static_cast<size_t>(lay.P) * sizeof(unsigned long long);
  static SmemLimit limit;
  const cudaError_t e = limit.ensure(reinterpret_cast<const void*>(pack_kernel),
                                     PCTREE_MAX_POOL * sizeof(unsigned long long));
  if (e != cudaSuccess) return e;
  pack_kernel<<<c.batch, kPackThreads, smem, stream>>>(
      c.B, c.k, c.N, lay.P, c.pos_offset,
      reinterpret_cast<const int32_t*>(ws + lay.off_pool_tok),
      reinterpret_cast<const int32_t*>(ws + lay.off_pool_par),
      reinterpret_cast<const float2*>(ws + lay.off_pool_s), out);
  return cudaGetLastError();
}

cudaError_t launch_accept(const pctree_config& c, const pctree_tree& tree,
                          const int32_t* target, int32_t* accepted_idx,
                          int32_t* accepted_len, int32_t* bonus,
                          cudaStream_t stream) {
  const int warps = 4;
  const int blocks = (c.batch + warps - 1) / warps;
  accept_kernel<<<blocks, warps * 32, 0, stream>>>(
      c.B, c.N, tree.n_nodes, tree.tokens, tree.parent, target, accepted_idx,
      accepted_len, bonus, c.batch);
  return cudaGetLastError();
}

}  // namespace pct
