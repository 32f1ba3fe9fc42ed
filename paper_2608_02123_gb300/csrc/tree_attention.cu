// pctree_tree_attention: one grouped-query attention layer of the target's
// tree-verification forward (Sec. 4.2; Appendix A "Tensor implementation"):
// every drafted node attends to the verified prefix, itself and its
// root-to-node ancestors.
//
// Work items: request r, KV head h, one or two query tiles (TILES) and a
// range of 64-key blocks.  A tile's rows are (node, query head of the group)
// pairs, node-major: row t = node_local * G + g, R = G * nodes_per_tile <=
// 128.  The G query heads sharing KV head h, and an item's tiles, read each
// K/V block once.  The kernel is persistent: one CTA per SM takes items in
// rounds of gridDim.x, forwards and backwards in turn, over a list ordered by
// decreasing request length (longest first keeps the last round short), so
// its set-up (barriers, TMEM) is paid once and the next item's loads and S
// products overlap the current item's last blocks and output.
//
//   warp 0      TMA producer: K and V blocks (64 keys x 128 dims, two 64-dim
//               halves each, 128-byte swizzle) into a ring (five stages for
//               one tile, four for two) that runs on across items
//   warp 1      S issuer: each item's Q tiles (once the previous item's S
//               products are done), then S_b = Q K_b^T per tile (tcgen05.mma,
//               M=128, N=64 keys, K=128 dims) into one of the tile's two TMEM
//               buffers, up to two blocks ahead of its softmax
//   warps 2..5  softmax and output of tile 0 (warps 6..9: tile 1): one thread
//               per TMEM lane = tile row; each S row is read from TMEM once,
//               masked and scaled; P = 2^(s - m_used) rounded to bf16 pairs is
//               written back over the first 32 columns of the S buffer (the
//               TMEM A operand of the second MMA).  O accumulates in TMEM
//               across an item's blocks; the
//               reference m_used rises (O and the row sum rescaled in place,
//               tcgen05.ld / st) only when a block's maximum exceeds it by
//               more than 8 in log2 units, so P stays below 2^8.  After the
//               item's last block the same warps normalise O and store it.
//   next warp   PV issuer: O += P_b V_b per tile (M=128, N=128 dims, K=64
//               keys; P read from TMEM, V the MN-major shared-memory operand,
//               dims contiguous) as soon as the tile's P_b is written; its
//               commit frees the S buffer and, after the item's tiles, the K/V
//               stage (S_b, the other reader, finished before P_b existed)
//   last warp   ancestor bits: the next item's ancestor-or-self masks (from
//               the packed parents) into the second of two buffers
//
// With two tiles each SM sub-partition runs one softmax warp of each, so one
// tile's waits overlap the other's arithmetic; TMEM then holds 2 x (two
// 64-column S buffers + a 128-column O) = 512 columns.  One tile per item is
// chosen when two-tile items would leave SMs idle.  Key blocks of a request may be split over several items (few
// requests, long prefixes); each then writes (max, sum, unnormalised O) of
// its rows and a second kernel merges the splits, spread over all SMs.  All
// waits are bounded (1 s) and end in PCTREE_ERR_TIMEOUT.
#include <cuda_bf16.h>

#include "pctree_common.cuh"
#include "sm103_ptx.cuh"

namespace pct {
namespace {

constexpr int kBK = 64;                   // keys per block
constexpr int kHalfBytes = 128 * 128;     // Q: 128 rows x 64 bf16 (one dim half)
constexpr int kQBytes = 2 * kHalfBytes;   // one Q tile
constexpr int kKVHalf = kBK * 128;        // K or V: 64 keys x 64 bf16 (one dim half)
constexpr int kStageBytes = 4 * kKVHalf;  // K (two halves) then V (two halves)
constexpr int kMaskWords = PCTREE_ATTN_MAX_N / 32;
constexpr uint64_t kAttnLimitNs = 1000000000ull;

constexpr int kMaxOrder = 256;            // requests ordered by length in shared memory

// Layout of a CTA with TILES query tiles (1 or 2): the Q tiles and a K/V
// ring in shared memory (five stages for one tile, four for two); per tile,
// two S buffers of 64 fp32 columns in TMEM (P, packed bf16 pairs, overwrites
// the first 32 columns of its S buffer and is the TMEM A operand of the PV
// product) and a 128-column O.
template <int TILES>
struct AttnCfg {
  static constexpr int kThreads = 32 * (4 + 4 * TILES);   // roles above
  static constexpr int kPVWarp = 2 + 4 * TILES;
  static constexpr int kAncWarp = 3 + 4 * TILES;
  static constexpr int kStages = TILES == 1 ? 5 : 4;
  static constexpr int kQOff = 0;
  static constexpr int kKVOff = TILES * kQBytes;
  static constexpr int kTailOff = kKVOff + kStages * kStageBytes;
  // TMEM: tile j's S buffer sb at columns (2j + sb) * kBK, its O (128
  // columns) at kOCol + 128 j
  static constexpr uint32_t kOCol = 2 * TILES * kBK;
  static constexpr uint32_t kTmemCols = kOCol + 128 * TILES <= 256 ? 256 : 512;
  static_assert(kOCol + 128 * TILES <= 512, "TMEM columns");
};

// Barriers count blocks over the CTA's whole item sequence: K/V stage g %
// kStages of the g-th block, S/P buffer g_j & 1 of the g_j-th block of tile
// j, ancestor buffer k & 1 of the k-th item.
template <int TILES>
struct AttnTail {
  static constexpr int kStages = AttnCfg<TILES>::kStages;
  uint64_t q_full, q_empty;
  uint64_t kv_full[kStages], kv_empty[kStages];
  uint64_t s_full[TILES][2];               // S written
  uint64_t p_full[TILES][2];               // P written over it
  uint64_t p_empty[TILES][2];              // PV product done: buffer free
  uint64_t anc_full[2], anc_empty[2];
  uint64_t done;
  uint32_t tmem_base;
  int abort;
  int last[TILES];
  uint32_t anc[2][TILES][128][kMaskWords];   // ancestor-or-self bits per node
  int32_t par[PCTREE_ATTN_MAX_N];            // packed parents being walked
  int32_t pre[kMaxOrder], nn[kMaxOrder];     // validated prefix / node counts
  int32_t order[kMaxOrder];                  // requests by decreasing key count
};

template <int TILES>
constexpr size_t attn_smem() {
  return AttnCfg<TILES>::kTailOff + sizeof(AttnTail<TILES>) + 1024;
}
static_assert(attn_smem<1>() <= 227 * 1024 && attn_smem<2>() <= 227 * 1024,
              "shared memory per CTA");

struct AttnArgs {
  const int32_t* prefix;
  const int32_t* n_nodes;
  const int32_t* parent;
  uint16_t* out;          // bf16 [batch][N][Hq][128]
  float* part_o;          // [unit][split][128][128]
  float2* part_ml;        // [unit][split][128]  (max in log2 units, sum)
  int32_t* status;
  int batch, N, Hq, Hkv, G, npt, R, nqt, tpc, npair, max_slots, n_split, bps;
  int items;              // batch * Hkv * npair * n_split
  float scale_log2;       // softmax scale * log2(e)
};

// One work item: request r, KV head kvh, query tiles qt0 .. qt0+ntile-1 and
// key blocks kb0 .. kb0+nblk-1 of the request's n_keys = Tp + n keys.
struct AttnItem {
  int r, kvh, qt0, ntile, split, Tp, n, n_keys, kb0, nblk;
};

// A request with an impossible prefix or tree size attends to nothing (its
// rows are written as 0 and the launch reports PCTREE_ERR_INVALID_ARG).
__device__ __forceinline__ bool request_ok(const AttnArgs& a, int Tp, int n) {
  return Tp >= 0 && n >= 0 && n <= a.N && static_cast<long long>(Tp) + n <= a.max_slots;
}

// Item `idx` of the item list: the items of request idx / per_req (of that
// rank in the longest-first order when `ranked`), as (split, KV head, tile
// pair) triples.  `staged`: the validated request sizes are in shared
// memory.
template <typename Tail>
__device__ __forceinline__ AttnItem item_facts(const AttnArgs& a, const Tail* T, int idx,
                                               bool ranked, bool staged) {
  AttnItem it;
  const int per_req = a.Hkv * a.npair * a.n_split;
  const int ri = idx / per_req, rest = idx - ri * per_req;
  it.r = ranked ? T->order[ri] : ri;
  it.split = rest / (a.Hkv * a.npair);
  it.kvh = (rest / a.npair) % a.Hkv;
  it.qt0 = (rest % a.npair) * a.tpc;
  it.ntile = min(a.tpc, a.nqt - it.qt0);
  if (staged) {
    it.Tp = T->pre[it.r];
    it.n = T->nn[it.r];
  } else {
    it.Tp = a.prefix[it.r];
    it.n = a.n_nodes[it.r];
    if (!request_ok(a, it.Tp, it.n)) it.Tp = it.n = 0;
  }
  it.n_keys = it.n > 0 ? it.Tp + it.n : 0;       // no queries: nothing to do
  const int nb_r = (it.n_keys + kBK - 1) / kBK;
  it.kb0 = it.split * a.bps;
  it.nblk = max(0, min(it.kb0 + a.bps, nb_r) - it.kb0);
  return it;
}

// Position in the longest-first list of this CTA's k-th item: rounds of
// gridDim.x items, taken forwards and backwards in turn, so every CTA gets a
// mix of long and short items.
__device__ __forceinline__ long long item_pos(int k) {
  const long long base = static_cast<long long>(k) * gridDim.x;
  return (k & 1) ? base + gridDim.x - 1 - blockIdx.x : base + blockIdx.x;
}

// 32 lanes x 8 columns of 32-bit TMEM words from registers: thread t of the
// warp writes lane (taddr.lane + t), columns taddr.col .. +7.
__device__ __forceinline__ void tmem_st_32x32b_x8(uint32_t taddr, const uint32_t (&r)[8]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
      : "memory");
}

// 32 lanes x 16 columns of 32-bit TMEM words from registers (see
// tmem_st_32x32b_x8).
__device__ __forceinline__ void tmem_st_32x32b_x16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15])
      : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem]: the A operand (M = 128 rows on the TMEM
// lanes, 16 K elements as 8 columns of bf16 pairs, the lower half holding the
// even element) is read from tensor memory.  Issued by one thread.
__device__ __forceinline__ void tc_mma_bf16_tmem_a(uint32_t d_tmem, uint32_t a_tmem,
                                                   uint64_t b_desc, uint32_t idesc,
                                                   uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Records the first error in the optional status word.
__device__ __forceinline__ void report(int32_t* status, int code) {
  if (status != nullptr) atomicCAS(status, 0, code);
}

// Allowed-key bits of 32 consecutive slots kc0 .. kc0+31 for a row whose
// node has ancestor-or-self bits `anc`: the whole prefix (slots < T) and
// the tree slots T + m of its ancestors (the bits are 0 past the tree).
__device__ __forceinline__ uint32_t allowed_bits(int kc0, int T,
                                                 const uint32_t* anc) {
  uint32_t bits = 0;
  const int pm = T - kc0;                       // prefix slots in the chunk
  if (pm >= 32) return 0xffffffffu;
  if (pm > 0) bits = (1u << pm) - 1u;
  const int m0 = kc0 - T;                       // tree index of slot kc0
  if (m0 >= 0) {
    const int w = m0 >> 5, sh = m0 & 31;
    uint32_t lo = w < kMaskWords ? anc[w] : 0u;
    uint32_t hi = (w + 1) < kMaskWords ? anc[w + 1] : 0u;
    bits |= sh == 0 ? lo : ((lo >> sh) | (hi << (32 - sh)));
  } else if (m0 > -32) {
    bits |= anc[0] << (-m0);
  }
  return bits;
}

template <int TILES>
__global__ void __launch_bounds__(AttnCfg<TILES>::kThreads, 1)
tree_attn_kernel(const __grid_constant__ CUtensorMap tm_q,
                 const __grid_constant__ CUtensorMap tm_k,
                 const __grid_constant__ CUtensorMap tm_v, AttnArgs a) {
  using C = AttnCfg<TILES>;
  constexpr int kStages = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  AttnTail<TILES>* T = reinterpret_cast<AttnTail<TILES>*>(sm + C::kTailOff);
  uint8_t* sq = sm + C::kQOff;
  // ring stage s: K (two dim halves) then V (two dim halves)
  auto kv_k = [&](int s) { return sm + C::kKVOff + s * kStageBytes; };
  auto kv_v = [&](int s) { return sm + C::kKVOff + s * kStageBytes + 2 * kKVHalf; };
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long n_items = a.items;
  // ancestor-or-self bits of an item's tile nodes into buffer ab (one warp:
  // stage the request's packed parents, then walk up from each node)
  auto ancestor_bits = [&](const AttnItem& it, int ab) {
    for (int i = lane; i < it.n; i += 32)
      T->par[i] = a.parent[static_cast<size_t>(it.r) * a.N + i];
    __syncwarp();
    for (int i = lane; i < it.ntile * a.npt; i += 32) {
      const int j = i / a.npt, nl = i - j * a.npt;
      uint32_t bits[kMaskWords];
#pragma unroll
      for (int w = 0; w < kMaskWords; ++w) bits[w] = 0u;
      int x = (it.qt0 + j) * a.npt + nl;
      for (int steps = 0; steps <= it.n && x >= 0 && x < it.n; ++steps) {
#pragma unroll
        for (int w = 0; w < kMaskWords; ++w)
          if ((x >> 5) == w) bits[w] |= 1u << (x & 31);
        const int px = T->par[x];
        x = px < x ? px : -1;          // parents precede children
      }
#pragma unroll
      for (int w = 0; w < kMaskWords; ++w) T->anc[ab][j][nl][w] = bits[w];
    }
    __syncwarp();                      // all lanes done with par and anc
  };
  // the longest-first order only matters when CTAs take several items; the
  // request sizes are then staged in shared memory too
  const bool ranked = a.batch <= kMaxOrder && n_items > static_cast<long long>(gridDim.x);
  const bool staged = ranked;
  // with one item per CTA its copies start right after the barrier set-up
  // (thread 0, the producer, issues Q and the first K/V blocks)
  int g_pre = 0;
  bool q_pre = false;

  // ---------------- set-up (once per CTA) ----------------
  if (threadIdx.x == 0) {
    mbar_init(&T->q_full, 1);
    mbar_init(&T->q_empty, 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&T->kv_full[s], 1);
      mbar_init(&T->kv_empty[s], 1);
    }
    for (int j = 0; j < TILES; ++j) {
      for (int sb = 0; sb < 2; ++sb) {
        mbar_init(&T->s_full[j][sb], 1);
        mbar_init(&T->p_full[j][sb], 4);
        mbar_init(&T->p_empty[j][sb], 1);
      }
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&T->anc_full[s], 1);
      mbar_init(&T->anc_empty[s], 4 * TILES);   // every softmax warp
    }
    mbar_init(&T->done, 2);              // one commit from each MMA issuer
    T->abort = 0;
    fence_barrier_init();
  }
  // programmatic dependent launch: the launch and the set-up above overlap
  // the previous kernel of the stream; every global access (request sizes,
  // Q, K, V, the output) comes after it is complete
  pdl_launch_dependents();
  pdl_wait();
  if (!ranked && (threadIdx.x == 0 || threadIdx.x == 32)) {
    const AttnItem it = item_facts(a, T, static_cast<int>(blockIdx.x), false, false);
    q_pre = it.nblk > 0;                 // known to the S issuer (thread 32) too
    if (threadIdx.x == 0 && it.nblk > 0) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
      mbar_arrive_expect_tx(&T->q_full, static_cast<uint32_t>(it.ntile) * 2u *
                                            static_cast<uint32_t>(a.R) * 128u);
      for (int j = 0; j < it.ntile; ++j) {
        const int node0 = (it.qt0 + j) * a.npt;
        tma_load_4d(sq + j * kQBytes, &tm_q, &T->q_full, 0, it.kvh * a.G, node0, it.r);
        tma_load_4d(sq + j * kQBytes + kHalfBytes, &tm_q, &T->q_full, 64, it.kvh * a.G, node0,
                    it.r);
      }
      for (; g_pre < min(kStages, it.nblk); ++g_pre) {
        const int s = g_pre, key0 = (it.kb0 + g_pre) * kBK;
        mbar_arrive_expect_tx(&T->kv_full[s], static_cast<uint32_t>(kStageBytes));
        tma_load_4d(kv_k(s), &tm_k, &T->kv_full[s], 0, it.kvh, key0, it.r);
        tma_load_4d(kv_k(s) + kKVHalf, &tm_k, &T->kv_full[s], 64, it.kvh, key0, it.r);
        tma_load_4d(kv_v(s), &tm_v, &T->kv_full[s], 0, it.kvh, key0, it.r);
        tma_load_4d(kv_v(s) + kKVHalf, &tm_v, &T->kv_full[s], 64, it.kvh, key0, it.r);
      }
    }
  }
  // requests: validated sizes (reported once) and, when ranked, staged and
  // ordered by key count
  if (staged || blockIdx.x == 0) {
    for (int u = threadIdx.x; u < a.batch; u += blockDim.x) {
      int Tp = a.prefix[u], n = a.n_nodes[u];
      if (!request_ok(a, Tp, n)) {
        if (blockIdx.x == 0) report(a.status, PCTREE_ERR_INVALID_ARG);
        Tp = n = 0;
      }
      if (staged) {
        T->pre[u] = Tp;
        T->nn[u] = n;
      }
    }
  }
  if (ranked) {
    __syncthreads();
    for (int u = threadIdx.x; u < a.batch; u += blockDim.x) {
      const int ku = T->nn[u] > 0 ? T->pre[u] + T->nn[u] : 0;
      int rank = 0;
      for (int v = 0; v < a.batch; ++v) {
        const int kv = T->nn[v] > 0 ? T->pre[v] + T->nn[v] : 0;
        rank += (kv > ku || (kv == ku && v < u)) ? 1 : 0;
      }
      T->order[rank] = u;
    }
  }
  // rows R..127 of each Q tile are never loaded: zero them once (read by
  // the MMA)
  const int zq = (128 - a.R) * 8;                  // 16-byte chunks per half
  for (int i = threadIdx.x; i < TILES * 2 * zq; i += blockDim.x) {
    const int j = i / (2 * zq), half = (i / zq) & 1, rem = i % zq;
    *reinterpret_cast<uint4*>(sq + j * kQBytes + half * kHalfBytes + (a.R + rem / 8) * 128 +
                              (rem % 8) * 16) = make_uint4(0, 0, 0, 0);
  }
  fence_proxy_async_smem();
  if (warp == 1) tmem_alloc(&T->tmem_base, C::kTmemCols);
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = T->tmem_base;
  volatile int* abort_v = &T->abort;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer: K and V blocks ----------------
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
      int g = 0;                                   // blocks issued
      bool ok = true;
      for (int k = 0; ok; ++k) {
        const long long pos = item_pos(k);
        if (pos >= n_items) break;
        const AttnItem it = item_facts(a, T, static_cast<int>(pos), ranked, staged);
        // blocks issued during the set-up (first item only)
        const int b0 = k == 0 ? g_pre : 0;
        g += b0;
        for (int b = b0; b < it.nblk; ++b, ++g) {
          const int s = g % kStages, key0 = (it.kb0 + b) * kBK;
          if (g >= kStages && !mbar_wait_bounded(&T->kv_empty[s], ((g / kStages) - 1) & 1,
                                                 abort_v, kAttnLimitNs)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&T->kv_full[s], static_cast<uint32_t>(kStageBytes));
          tma_load_4d(kv_k(s), &tm_k, &T->kv_full[s], 0, it.kvh, key0, it.r);
          tma_load_4d(kv_k(s) + kKVHalf, &tm_k, &T->kv_full[s], 64, it.kvh, key0, it.r);
          tma_load_4d(kv_v(s), &tm_v, &T->kv_full[s], 0, it.kvh, key0, it.r);
          tma_load_4d(kv_v(s) + kKVHalf, &tm_v, &T->kv_full[s], 64, it.kvh, key0, it.r);
        }
      }
      if (!ok) {
        *abort_v = 1;
        report(a.status, PCTREE_ERR_TIMEOUT);
      }
      // copies still in flight land before the CTA may exit
      for (int b = g - kStages > 0 ? g - kStages : 0; b < g; ++b)
        (void)mbar_wait_bounded(&T->kv_full[b % kStages], (b / kStages) & 1, abort_v,
                                kAttnLimitNs);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- S issuer (and the Q tiles of each item) ----------------
      constexpr uint32_t idS = idesc_bf16_f32(128, kBK);
      tma_prefetch_desc(&tm_q);
      int g = 0, gj[TILES], q = 0;                 // blocks, per tile, Q loads
      for (int j = 0; j < TILES; ++j) gj[j] = 0;
      bool ok = true;
      for (int k = 0; ok; ++k) {
        const long long pos = item_pos(k);
        if (pos >= n_items) break;
        const AttnItem it = item_facts(a, T, static_cast<int>(pos), ranked, staged);
        if (it.nblk == 0) continue;
        // the Q buffers are free once the previous item's S products are done
        if (q > 0 && !mbar_wait_bounded(&T->q_empty, (q - 1) & 1, abort_v, kAttnLimitNs)) {
          ok = false;
          break;
        }
        if (!(q == 0 && q_pre)) {          // else issued during the set-up
          mbar_arrive_expect_tx(&T->q_full, static_cast<uint32_t>(it.ntile) * 2u *
                                                static_cast<uint32_t>(a.R) * 128u);
          for (int j = 0; j < it.ntile; ++j) {
            const int node0 = (it.qt0 + j) * a.npt;
            tma_load_4d(sq + j * kQBytes, &tm_q, &T->q_full, 0, it.kvh * a.G, node0, it.r);
            tma_load_4d(sq + j * kQBytes + kHalfBytes, &tm_q, &T->q_full, 64, it.kvh * a.G,
                        node0, it.r);
          }
        }
        if (!mbar_wait_bounded(&T->q_full, q & 1, abort_v, kAttnLimitNs)) {
          ok = false;
          break;
        }
        ++q;
        const uint32_t q0 = smem_u32(sq);
        for (int b = 0; ok && b < it.nblk; ++b, ++g) {
          const int s = g % kStages;
          ok = mbar_wait_bounded(&T->kv_full[s], (g / kStages) & 1, abort_v, kAttnLimitNs);
          const uint32_t k0 = smem_u32(kv_k(s));
          for (int j = 0; ok && j < it.ntile; ++j) {
            const int sb = gj[j] & 1;
            // tile j's S buffer sb holds the P of block gj - 2 until that
            // block's PV product is done
            if (gj[j] >= 2 && !mbar_wait_bounded(&T->p_empty[j][sb], ((gj[j] >> 1) - 1) & 1,
                                                 abort_v, kAttnLimitNs)) {
              ok = false;
              break;
            }
            tc_fence_after_sync();
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {      // 128 dims in steps of 16
              tc_mma_bf16(tmem + (2 * j + sb) * kBK,
                          desc_kmajor_sw128(q0 + j * kQBytes + (kk >> 2) * kHalfBytes +
                                            (kk & 3) * 32),
                          desc_kmajor_sw128(k0 + (kk >> 2) * kKVHalf + (kk & 3) * 32), idS,
                          kk > 0 ? 1u : 0u);
            }
            tc_commit(&T->s_full[j][sb]);
            ++gj[j];
          }
        }
        tc_commit(&T->q_empty);          // arrives once the item's S products are done
      }
      if (!ok) {
        *abort_v = 1;
        report(a.status, PCTREE_ERR_TIMEOUT);
      }
      tc_commit(&T->done);               // every MMA this thread issued has finished
      (void)mbar_wait_bounded(&T->done, 0, abort_v, kAttnLimitNs);
    }
  } else if (warp == C::kPVWarp) {
    if (lane == 0) {
      // ---------------- PV issuer ----------------
      constexpr uint32_t idO = idesc_bf16_f32_bmn(128, 128);
      int g = 0, gj[TILES];
      for (int j = 0; j < TILES; ++j) gj[j] = 0;
      bool ok = true;
      for (int k = 0; ok; ++k) {
        const long long pos = item_pos(k);
        if (pos >= n_items) break;
        const AttnItem it = item_facts(a, T, static_cast<int>(pos), ranked, staged);
        for (int b = 0; ok && b < it.nblk; ++b, ++g) {
          const int s = g % kStages;
          const uint32_t v0 = smem_u32(kv_v(s));
          for (int j = 0; j < it.ntile; ++j) {
            const int sb = gj[j] & 1;
            // P_b of tile j, and with it S_b, is complete
            if (!mbar_wait_bounded(&T->p_full[j][sb], (gj[j] >> 1) & 1, abort_v,
                                   kAttnLimitNs)) {
              ok = false;
              break;
            }
            tc_fence_after_sync();
            const uint32_t pa = tmem + (2 * j + sb) * kBK;       // P: 32 columns
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk) {
              // A: 16 keys of P = 8 TMEM columns; B: 16 keys = 16 rows of 128 B
              // of V, the dims 64..127 half kKVHalf further on
              tc_mma_bf16_tmem_a(tmem + C::kOCol + j * 128, pa + kk * 8,
                                 desc_mnmajor_sw128(v0 + kk * 16 * 128, kKVHalf, 1024), idO,
                                 (b > 0 || kk > 0) ? 1u : 0u);   // O accumulates over the item
            }
            tc_commit(&T->p_empty[j][sb]);
            ++gj[j];
          }
          // the item's S and PV products of this block have read the stage
          if (ok) tc_commit(&T->kv_empty[s]);
        }
      }
      if (!ok) {
        *abort_v = 1;
        report(a.status, PCTREE_ERR_TIMEOUT);
      }
      tc_commit(&T->done);
      (void)mbar_wait_bounded(&T->done, 0, abort_v, kAttnLimitNs);
    }
  } else if (warp == C::kAncWarp) {
    // ---------------- ancestor bits of each item, one item ahead ----------------
    for (int k = 0;; ++k) {
      const long long pos = item_pos(k);
      if (pos >= n_items) break;
      const AttnItem it = item_facts(a, T, static_cast<int>(pos), ranked, staged);
      const int ab = k & 1;
      // buffer ab was last read by the softmax warps for item k - 2
      const bool got = k < 2 || mbar_wait_bounded(&T->anc_empty[ab], ((k >> 1) - 1) & 1,
                                                   abort_v, kAttnLimitNs);
      if (!__all_sync(kFull, got)) {
        if (lane == 0) {
          *abort_v = 1;
          report(a.status, PCTREE_ERR_TIMEOUT);
        }
        break;
      }
      ancestor_bits(it, ab);
      if (lane == 0) mbar_arrive(&T->anc_full[ab]);
    }
  }
  else if (warp >= 2 && warp < 2 + 4 * TILES) {
    // ---------------- softmax and output, one thread per tile row ----------------
    // O accumulates in TMEM through the PV MMA with P = 2^(s - m_used); the
    // reference m_used moves (and O and l are rescaled in place) only when
    // a block's maximum exceeds it by more than 2^8, so P stays <= 256.
    const int j = (warp - 2) / 4;            // the tile of this warp
    const int quad = warp & 3;               // TMEM lanes quad*32 .. +31
    const int t = quad * 32 + lane;          // tile row
    const int nl = t / a.G, g = t - nl * a.G;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const uint32_t s_col = lane_base + 2 * j * kBK, o_col = lane_base + C::kOCol + j * 128;
    const float sc = a.scale_log2;
    // the warp continues only if all its lanes saw the phase complete, so
    // the warp-collective tcgen05 loads that follow never diverge
    auto wwait = [&](uint64_t* bar, uint32_t parity) -> bool {
      const bool got = mbar_wait_bounded(bar, parity, abort_v, kAttnLimitNs);
      return __all_sync(kFull, got);
    };
    int gr = 0, gj = 0;                      // blocks of the ring, of tile j
    for (int k = 0;; ++k) {
      const long long pos = item_pos(k);
      if (pos >= n_items) break;
      const AttnItem it = item_facts(a, T, static_cast<int>(pos), ranked, staged);
      const int ab = k & 1;
      // the item's ancestor bits; both tiles' warps take part in the buffer
      // hand-off, also for an item without a tile j
      bool ok = wwait(&T->anc_full[ab], (k >> 1) & 1);
      const bool active = j < it.ntile;
      const int node = (it.qt0 + j) * a.npt + nl;
      const bool row_ok = active && t < a.R && node < it.n;
      const uint32_t* anc = T->anc[ab][j][nl < a.npt ? nl : 0];
      const int Tp = it.Tp, n_keys = it.n_keys, nblk = active ? it.nblk : 0;
      const int g0 = gj;                     // the item's first block of tile j
      float m_used = -INFINITY, l_sum = 0.0f;  // O and l_sum are relative to m_used
      for (int b = 0; ok && b < nblk; ++b) {
        const int gb = g0 + b, sb = gb & 1, st = (gr + b) % kStages;
        const int key0 = (it.kb0 + b) * kBK;
        if (!wwait(&T->s_full[j][sb], (gb >> 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        float x[kBK];
        {
          uint32_t* xu = reinterpret_cast<uint32_t*>(x);
#pragma unroll
          for (int c = 0; c < kBK / 32; ++c)
            tmem_ld_32x32b_x32(s_col + sb * kBK + c * 32,
                               *reinterpret_cast<uint32_t(*)[32]>(xu + c * 32));
          tmem_ld_wait();
        }
        // scaled scores; keys the row may not see become -inf (eight
        // independent running maxima keep the dependency chains short)
        float m8[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) m8[u] = -INFINITY;
        if (row_ok && key0 + kBK <= Tp) {      // a block of prefix keys only
#pragma unroll
          for (int k2 = 0; k2 < kBK; ++k2) {
            x[k2] *= sc;
            m8[k2 & 7] = fmaxf(m8[k2 & 7], x[k2]);
          }
        } else {
#pragma unroll
          for (int c = 0; c < kBK / 32; ++c) {
            const uint32_t al = row_ok ? allowed_bits(key0 + c * 32, Tp, anc) : 0u;
#pragma unroll
            for (int k2 = 0; k2 < 32; ++k2) {
              const float v = ((al >> k2) & 1u) ? x[c * 32 + k2] * sc : -INFINITY;
              x[c * 32 + k2] = v;
              m8[k2 & 7] = fmaxf(m8[k2 & 7], v);
            }
          }
        }
        const float mx = fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])),
                               fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7])));
        // the last block of the request: V rows past the tree hold whatever
        // the cache held there; zero them so that 0 * (non-finite) cannot
        // reach O.  Both tiles' warps do it: each tile's PV product then reads
        // rows its own warps zeroed and fenced, and the other tile only ever
        // writes the same zero bytes there.
        const int valid = n_keys - key0;
        if (valid < kBK) {
          if (!wwait(&T->kv_full[st], ((gr + b) / kStages) & 1)) {
            ok = false;
            break;
          }
          uint8_t* v = kv_v(st);
          for (int i = t; i < 2 * (kBK - valid) * 8; i += 128) {
            const int half = i / ((kBK - valid) * 8), rem = i % ((kBK - valid) * 8);
            *reinterpret_cast<uint4*>(v + half * kKVHalf + (valid + rem / 8) * 128 +
                                      (rem % 8) * 16) = make_uint4(0, 0, 0, 0);
          }
        }
        // move the reference up where a row needs it; tcgen05.ld / st are
        // warp-collective, so the warp rescales together (alpha = 1 for rows
        // that keep their reference)
        const bool mine = mx > m_used + 8.0f;
        const float alpha = mine ? ex2_approx(m_used - mx) : 1.0f;   // 0 from -inf
        if (__any_sync(kFull, mine)) {
          if (b >= 1) {
            // O must hold every block before b: the PV product of block b - 1
            // has finished
            if (!wwait(&T->p_empty[j][(gb - 1) & 1], ((gb - 1) >> 1) & 1)) {
              ok = false;
              break;
            }
            tc_fence_after_sync();
            // eight columns at a time: the block's scores stay live meanwhile
#pragma unroll 4
            for (int c = 0; c < 16; ++c) {
              uint32_t y[8];
              tmem_ld_32x32b_x8(o_col + c * 8, y);
              tmem_ld_wait();
#pragma unroll
              for (int k2 = 0; k2 < 8; ++k2)
                y[k2] = __float_as_uint(__uint_as_float(y[k2]) * alpha);
              tmem_st_32x32b_x8(o_col + c * 8, y);
            }
            tmem_st_wait();
          }
          if (mine) {
            l_sum *= alpha;
            m_used = mx;
          }
        }
        // P = 2^(s - m_used) in bf16 pairs over the first 32 columns of the
        // S buffer (all of S is in registers): the TMEM A operand of the PV
        // MMA
        const float mref = m_used == -INFINITY ? 0.0f : m_used;
        float ls[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
        for (int c = 0; c < kBK / 32; ++c) {
          uint32_t pk[16];
#pragma unroll
          for (int h = 0; h < 16; ++h) {
            const float p0 = ex2_approx(x[c * 32 + 2 * h] - mref);
            const float p1 = ex2_approx(x[c * 32 + 2 * h + 1] - mref);
            ls[h & 3] += p0 + p1;
            const __nv_bfloat162 pb = __floats2bfloat162_rn(p0, p1);
            pk[h] = *reinterpret_cast<const uint32_t*>(&pb);
          }
          tmem_st_32x32b_x16(s_col + sb * kBK + c * 16, pk);
        }
        tmem_st_wait();
        l_sum += (ls[0] + ls[1]) + (ls[2] + ls[3]);
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(&T->p_full[j][sb]);
      }
      // the ancestor bits of this item are no longer needed
      __syncwarp();
      if (lane == 0) mbar_arrive(&T->anc_empty[ab]);
      // every PV product of the item has finished: the last one on each S/P
      // buffer (earlier ones are known complete)
      for (int gb = g0 + nblk - 2 > g0 ? g0 + nblk - 2 : g0; ok && gb < g0 + nblk; ++gb)
        if (!wwait(&T->p_empty[j][gb & 1], (gb >> 1) & 1)) ok = false;
      gr += it.nblk;
      gj += nblk;
      if (!ok) {
        *abort_v = 1;
        report(a.status, PCTREE_ERR_TIMEOUT);
      }
      // one decision for the tile's four softmax warps (they meet at named
      // barriers, which must see every one of them)
      named_barrier(1 + j, 128);
      if (t == 0) T->last[j] = *abort_v;
      named_barrier(1 + j, 128);
      ok = T->last[j] == 0;
      named_barrier(1 + j, 128);
      if (!ok) break;
      if (!active) continue;
      tc_fence_after_sync();
      // ---------------- output ----------------
      // O is read from TMEM in four 32-column chunks; tcgen05.ld is
      // warp-collective, so every lane loads and only valid rows store.  The
      // loads finish (tcgen05.wait::ld) before this warp's next P is
      // published, so the next item's first PV product cannot overwrite O
      // early.
      const int unit = (it.r * a.Hkv + it.kvh) * a.nqt + it.qt0 + j;
      const bool store_row = t < a.R && node < a.N;
      uint16_t* orow =
          a.out + ((static_cast<size_t>(it.r) * a.N + node) * a.Hq + it.kvh * a.G + g) * 128;
      auto store_chunk = [&](int c, const float (&v)[32], float inv) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint32_t w[4];
#pragma unroll
          for (int h = 0; h < 4; ++h) {
            const __nv_bfloat162 b2 =
                __floats2bfloat162_rn(v[q * 8 + 2 * h] * inv, v[q * 8 + 2 * h + 1] * inv);
            w[h] = *reinterpret_cast<const uint32_t*>(&b2);
          }
          *reinterpret_cast<uint4*>(orow + c * 32 + q * 8) = make_uint4(w[0], w[1], w[2], w[3]);
        }
      };
      auto load_chunk = [&](int c, float (&v)[32]) {
        if (nblk > 0) {
          uint32_t y[32];
          tmem_ld_32x32b_x32(o_col + c * 32, y);
          tmem_ld_wait();
#pragma unroll
          for (int k2 = 0; k2 < 32; ++k2) v[k2] = __uint_as_float(y[k2]);
        } else {
#pragma unroll
          for (int k2 = 0; k2 < 32; ++k2) v[k2] = 0.0f;
        }
      };
      if (a.n_split == 1) {
        const float inv = l_sum > 0.0f ? 1.0f / l_sum : 0.0f;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          float v[32];
          load_chunk(c, v);
          if (store_row) store_chunk(c, v, inv);
        }
      } else {
        const size_t slot = static_cast<size_t>(unit) * a.n_split + it.split;
        a.part_ml[slot * 128 + t] = make_float2(l_sum > 0.0f ? m_used : -INFINITY, l_sum);
        float4* po = reinterpret_cast<float4*>(a.part_o + (slot * 128 + t) * 128);
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          float v[32];
          load_chunk(c, v);
          if (l_sum > 0.0f) {
#pragma unroll
            for (int q = 0; q < 8; ++q)
              po[c * 8 + q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          }
        }
      }
      tc_fence_before_sync();
    }
  }
  // ---------------- teardown ----------------
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}
// Merges the key splits of every (request, KV head, tile) unit: one thread
// per 16 output dims of a row, 16 rows per CTA.  Per row the splits' maxima
// and sums give weights 2^(m_s - m*); the weighted partial outputs are summed
// four splits at a time (their loads in flight together) and normalised.
constexpr int kMergeThreads = 128;
constexpr int kMergeRows = 16;

__global__ void __launch_bounds__(kMergeThreads)
tree_attn_merge_kernel(AttnArgs a) {
  // launched while the attention kernel finishes: its partials are read
  // after it is complete
  pdl_launch_dependents();
  pdl_wait();
  const int unit = blockIdx.x;
  const int row = blockIdx.y * kMergeRows + (threadIdx.x >> 3);   // tile row
  const int d0 = (threadIdx.x & 7) * 16;
  const int qt = unit % a.nqt;
  const int kvh = (unit / a.nqt) % a.Hkv;
  const int r = unit / (a.nqt * a.Hkv);
  const int nl = row / a.G, g = row - nl * a.G;
  const int node = qt * a.npt + nl;
  if (row >= a.R || node >= a.N) return;
  const float2* ml = a.part_ml + static_cast<size_t>(unit) * a.n_split * 128 + row;
  float mstar = -INFINITY, lsum = 0.0f;
  for (int s0 = 0; s0 < a.n_split; s0 += 8) {   // eight loads in flight
    float2 v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u)
      v[u] = s0 + u < a.n_split ? ml[static_cast<size_t>(s0 + u) * 128]
                                : make_float2(-INFINITY, 0.0f);
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (v[u].y > 0.0f) mstar = fmaxf(mstar, v[u].x);
  }
  float acc[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) acc[j] = 0.0f;
  for (int s0 = 0; s0 < a.n_split; s0 += 4) {
    float4 v[4][4];
    float f[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      f[u] = 0.0f;
      if (s0 + u < a.n_split) {
        const float2 w = ml[static_cast<size_t>(s0 + u) * 128];
        if (w.y > 0.0f) {
          f[u] = exp2f(w.x - mstar);
          lsum = fmaf(w.y, f[u], lsum);
          const float4* src = reinterpret_cast<const float4*>(
              a.part_o + ((static_cast<size_t>(unit) * a.n_split + s0 + u) * 128 + row) * 128 + d0);
#pragma unroll
          for (int q = 0; q < 4; ++q) v[u][q] = src[q];
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (f[u] != 0.0f) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          acc[4 * q] = fmaf(v[u][q].x, f[u], acc[4 * q]);
          acc[4 * q + 1] = fmaf(v[u][q].y, f[u], acc[4 * q + 1]);
          acc[4 * q + 2] = fmaf(v[u][q].z, f[u], acc[4 * q + 2]);
          acc[4 * q + 3] = fmaf(v[u][q].w, f[u], acc[4 * q + 3]);
        }
      }
    }
  }
  const float inv = lsum > 0.0f ? 1.0f / lsum : 0.0f;
  uint16_t* orow = a.out + ((static_cast<size_t>(r) * a.N + node) * a.Hq + kvh * a.G + g) * 128 + d0;
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    uint32_t w[4];
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      const __nv_bfloat162 b2 =
          __floats2bfloat162_rn(acc[q * 8 + 2 * h] * inv, acc[q * 8 + 2 * h + 1] * inv);
      w[h] = *reinterpret_cast<const uint32_t*>(&b2);
    }
    *reinterpret_cast<uint4*>(orow + q * 8) = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

}  // namespace
}  // namespace pct

namespace pct {
namespace {

// Tiling of a configuration: query tiles per (request, KV head), tiles per
// item and the split of each request's key blocks over items.  Splits are
// chosen so that there are about as many items as the 152 SMs of a GB300
// when there are few (request, KV head, tile) units; they depend only on the
// configuration, so the workspace size does too.
struct AttnGeom {
  int G, npt, R, nqt, tpc, npair, nb_max, n_split, bps;
  long long units;                    // (request, KV head, query tile) triples
};

AttnGeom attn_geom(const pctree_attn_config& c) {
  AttnGeom g{};
  g.G = c.Hq / c.Hkv;
  g.npt = 128 / g.G < c.N ? 128 / g.G : c.N;
  g.R = g.G * g.npt;
  g.nqt = (c.N + g.npt - 1) / g.npt;
  // two tiles per item once such items still fill every SM (their softmax
  // waits overlap); otherwise one tile per item keeps more SMs busy
  const long long pairs = static_cast<long long>(c.batch) * c.Hkv * ((g.nqt + 1) / 2);
  g.tpc = (g.nqt >= 2 && pairs >= 152) ? 2 : 1;
  g.npair = (g.nqt + g.tpc - 1) / g.tpc;
  g.units = static_cast<long long>(c.batch) * c.Hkv * g.nqt;
  g.nb_max = (c.max_slots + kBK - 1) / kBK;
  const long long ctas = static_cast<long long>(c.batch) * c.Hkv * g.npair;
  long long want = (152 + ctas - 1) / ctas;
  if (want > g.nb_max) want = g.nb_max;
  if (want < 1) want = 1;
  g.bps = static_cast<int>((g.nb_max + want - 1) / want);
  g.n_split = (g.nb_max + g.bps - 1) / g.bps;
  return g;
}

pctree_status attn_check(const pctree_attn_config* c) {
  if (c == nullptr) return PCTREE_ERR_INVALID_ARG;
  if (c->batch < 1 || c->N < 1 || c->Hq < 1 || c->Hkv < 1 || c->D < 1 ||
      c->max_slots < c->N || !(c->scale > 0.0f) || !(c->scale < 1e30f))
    return PCTREE_ERR_INVALID_ARG;
  if (c->Hq % c->Hkv != 0) return PCTREE_ERR_INVALID_ARG;
  if (c->D != 128 || c->Hq / c->Hkv > 128 || c->N > PCTREE_ATTN_MAX_N ||
      c->batch > 65535 || c->Hkv > 65535)
    return PCTREE_ERR_UNSUPPORTED;
  const AttnGeom g = attn_geom(*c);
  if (static_cast<long long>(c->batch) * c->Hkv * g.npair * g.n_split > 0x7fffffffll)
    return PCTREE_ERR_UNSUPPORTED;
  return PCTREE_OK;
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

struct AttnWs {
  size_t part_o, part_ml, total;
};

AttnWs attn_ws(const pctree_attn_config& c, const AttnGeom& g) {
  AttnWs w{};
  if (g.n_split <= 1) return w;
  const size_t slots = static_cast<size_t>(g.units) * g.n_split * 128;
  w.part_o = 0;
  w.part_ml = align256(w.part_o + slots * 128 * sizeof(float));
  w.total = align256(w.part_ml + slots * sizeof(float2));
  return w;
}

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace pct

extern "C" {

size_t pctree_tree_attention_workspace_bytes(const pctree_attn_config* cfg) {
  if (pct::attn_check(cfg) != PCTREE_OK) return 0;
  return pct::attn_ws(*cfg, pct::attn_geom(*cfg)).total;
}

pctree_status pctree_tree_attention(const pctree_attn_config* cfg, const void* q,
                                    const void* k_cache, const void* v_cache,
                                    const int32_t* prefix_len,
                                    const int32_t* n_nodes, const int32_t* parent,
                                    void* out, void* workspace,
                                    size_t workspace_bytes, int32_t* status,
                                    void* stream_ptr) {
  pct::NvtxRange range("pctree_tree_attention");
  using namespace pct;
  pctree_status st = attn_check(cfg);
  if (st != PCTREE_OK) return st;
  const pctree_attn_config& c = *cfg;
  if (q == nullptr || k_cache == nullptr || v_cache == nullptr ||
      prefix_len == nullptr || n_nodes == nullptr || parent == nullptr ||
      out == nullptr || !al16(q) || !al16(k_cache) || !al16(v_cache) || !al16(out))
    return PCTREE_ERR_INVALID_ARG;
  const AttnGeom g = attn_geom(c);
  const AttnWs w = attn_ws(c, g);
  if (w.total > 0 && (workspace == nullptr || workspace_bytes < w.total ||
                      (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0))
    return PCTREE_ERR_WORKSPACE;
  int num_sms = 0;
  st = device_facts(&num_sms);
  if (st != PCTREE_OK) return st;
  CUtensorMap tm_q, tm_k, tm_v;
  const uint64_t hd = 128 * 2;                       // bytes of one head row
  {
    const uint64_t dims[4] = {128, static_cast<uint64_t>(c.Hq),
                              static_cast<uint64_t>(c.N), static_cast<uint64_t>(c.batch)};
    const uint64_t str[3] = {hd, hd * c.Hq, hd * c.Hq * c.N};
    const uint32_t box[4] = {64, static_cast<uint32_t>(g.G), static_cast<uint32_t>(g.npt), 1};
    st = encode_bf16_map_nd(&tm_q, q, 4, dims, str, box);
    if (st != PCTREE_OK) return st;
  }
  {
    const uint64_t dims[4] = {128, static_cast<uint64_t>(c.Hkv),
                              static_cast<uint64_t>(c.max_slots),
                              static_cast<uint64_t>(c.batch)};
    const uint64_t str[3] = {hd, hd * c.Hkv, hd * c.Hkv * c.max_slots};
    const uint32_t box[4] = {64, 1, static_cast<uint32_t>(kBK), 1};
    st = encode_bf16_map_nd(&tm_k, k_cache, 4, dims, str, box);
    if (st != PCTREE_OK) return st;
    st = encode_bf16_map_nd(&tm_v, v_cache, 4, dims, str, box);
    if (st != PCTREE_OK) return st;
  }
  cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);
  AttnArgs a{};
  a.prefix = prefix_len;
  a.n_nodes = n_nodes;
  a.parent = parent;
  a.out = static_cast<uint16_t*>(out);
  a.status = status;
  a.batch = c.batch;
  a.N = c.N;
  a.Hq = c.Hq;
  a.Hkv = c.Hkv;
  a.G = g.G;
  a.npt = g.npt;
  a.R = g.R;
  a.nqt = g.nqt;
  a.tpc = g.tpc;
  a.npair = g.npair;
  a.items = static_cast<int>(static_cast<long long>(c.batch) * c.Hkv * g.npair * g.n_split);
  a.max_slots = c.max_slots;
  a.n_split = g.n_split;
  a.bps = g.bps;
  a.scale_log2 = static_cast<float>(static_cast<double>(c.scale) * 1.4426950408889634);
  if (w.total > 0) {
    unsigned char* ws = static_cast<unsigned char*>(workspace);
    a.part_o = reinterpret_cast<float*>(ws + w.part_o);
    a.part_ml = reinterpret_cast<float2*>(ws + w.part_ml);
  }
  // a dummy status word is not needed: kernels test for NULL
  static SmemLimit limit1, limit2;
  if (limit1.ensure(reinterpret_cast<const void*>(tree_attn_kernel<1>), attn_smem<1>()) !=
          cudaSuccess ||
      limit2.ensure(reinterpret_cast<const void*>(tree_attn_kernel<2>), attn_smem<2>()) !=
          cudaSuccess)
    return PCTREE_ERR_CUDA;
  // persistent: one CTA per SM walks its share of the items; both kernels
  // are launched with programmatic stream serialization (each waits for its
  // predecessor before touching global memory)
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(static_cast<unsigned>(a.items < num_sms ? a.items : num_sms));
  lc.stream = stream;
  lc.attrs = attr;
  lc.numAttrs = 1;
  cudaError_t e;
  if (g.tpc == 2) {
    lc.blockDim = dim3(AttnCfg<2>::kThreads);
    lc.dynamicSmemBytes = attn_smem<2>();
    e = cudaLaunchKernelEx(&lc, tree_attn_kernel<2>, tm_q, tm_k, tm_v, a);
  } else {
    lc.blockDim = dim3(AttnCfg<1>::kThreads);
    lc.dynamicSmemBytes = attn_smem<1>();
    e = cudaLaunchKernelEx(&lc, tree_attn_kernel<1>, tm_q, tm_k, tm_v, a);
  }
  if (e != cudaSuccess) return PCTREE_ERR_CUDA;
  if (g.n_split > 1) {
    lc.gridDim = dim3(static_cast<unsigned>(g.units), (g.R + kMergeRows - 1) / kMergeRows);
    lc.blockDim = dim3(kMergeThreads);
    lc.dynamicSmemBytes = 0;
    if (cudaLaunchKernelEx(&lc, tree_attn_merge_kernel, a) != cudaSuccess) return PCTREE_ERR_CUDA;
  }
  return PCTREE_OK;
}

}  // extern "C"
