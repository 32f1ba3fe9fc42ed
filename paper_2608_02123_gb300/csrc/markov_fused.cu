// Markov projection of one PCTree stage with the stage's log-softmax
// normaliser and per-parent top-k folded into the epilogue (Eqs. 2-3), for
// bf16 heads and any number of Markov rows (the batched serving rounds):
//
//   z[row][v] = L_d[req(row)][v] + sum_h W_out[v][h] * X[row][h]
//
// is formed tile by tile in tensor memory and never written to HBM.  For
// every parent row the CTA keeps, over the vocabulary tiles it owns, a
// running (max, sum of exp) and a sorted top-k list of (z, token); at the end
// of the pass it publishes them as one partial per (row, CTA), which the
// stage's merge combines into the row's normaliser and children.
//
// Layout of the work: persistent CTAs (one per SM) take vocabulary tiles of
// 128 rows round-robin.  Warp 0 streams W_out tiles (MMA A, 128 x 64 bf16
// boxes, L2 evict_first) and the pass's parent rows (MMA B, NC x 64) with TMA
// into a shared-memory ring; warp 1 issues tcgen05.mma (M = 128 vocabulary
// rows, N = NC parent rows, f32 accumulators in TMEM, two buffers so the
// epilogue of one tile overlaps the MMAs of the next).  Warps 2..9 are the
// epilogue.  Per 64-column chunk of the accumulator:
//   A  each warp reads 32 TMEM lanes (its quadrant) x 32 columns with
//      tcgen05.ld and writes them transposed into shared memory, so that
//      one parent row's 128 logits of the tile lie contiguous;
//   B  each warp takes 8 of the chunk's parent rows: per row, a float4 of
//      logits per lane plus the base logits, a warp (max, sum-exp) folded
//      into the row's running pair, and the row's top-k list updated with
//      the logits that beat its current k-th entry (most tiles have none).
// A CTA's first tile seeds each row's list with a sort of the lanes' best
// logits.  The CTAs also share, per row, the best k-th list entry any of
// them holds (a 64-bit word in global memory raised with atomicMax after each
// tile): a logit below it is beaten by k logits of that CTA's slice alone,
// so it cannot be one of the row's k children and is not inserted.  The
// shared value only removes candidates that lose anyway, so the merged
// children do not depend on when a CTA reads it.  Rows are always handled
// by the same warp in the same tile order.
#include <cuda_runtime.h>

#include "pctree_common.cuh"
#include "sm103_ptx.cuh"

namespace pct {
namespace {

constexpr int kBM = 128;          // vocabulary rows per tile (MMA M)
constexpr int kBK = 64;           // K elements per ring slot (128 B of bf16)
constexpr int kUmmaK = 16;        // K per tcgen05.mma kind::f16
constexpr int kEpiWarps = 8;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kThreads = 64 + kEpiThreads;
constexpr int kCC = 64;           // accumulator columns per transpose chunk
constexpr int kRowsPerWarp = kCC / kEpiWarps;
constexpr int kCand = 16;         // compacted candidates per row and round
constexpr int kRegList = 16;      // k up to this: a row's list in registers
// the register lists are spread four lanes per row, four entries per lane
static_assert(kRowsPerWarp * 4 == 32 && kRegList == 4 * 4,
              "four lanes per row and four entries per lane");
constexpr int kMaxStages = 8;
constexpr int kSmemLimit = 227 * 1024;
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // 1 s per bounded wait
constexpr float kNegInf = -INFINITY;
constexpr float kPosInf = INFINITY;
constexpr float kLog2e = 1.4426950408889634f;

// Shared-memory plan of one instance (NC columns, k up to PCTREE_MAX_K).
template <int NC>
struct FusedProj {
  static constexpr int kABytes = kBM * kBK * 2;          // 16 KB
  static constexpr int kBBytes = NC * kBK * 2;           // 2..32 KB
  static constexpr int kStageBytes = kABytes + kBBytes;  // multiple of 1024
  // accumulator buffers: as many as the 512 TMEM columns hold, up to 4, so
  // the MMAs run ahead of a slow epilogue tile
  static constexpr int kAccBufs = 512 / NC > 4 ? 4 : 512 / NC;
  static constexpr int kTmemCols = kAccBufs * NC < 32 ? 32 : kAccBufs * NC;
  static constexpr size_t kZBytes = static_cast<size_t>(kCC) * kBM * sizeof(float);
  // per-row running max and sum of exp, and the k-th entry of the row's
  // top-k list (the insertion threshold)
  static constexpr size_t kRowBytes = static_cast<size_t>(NC) * 12;
  static constexpr size_t kBarBytes = 256;
  // per epilogue warp, per row of a chunk: kCand compacted candidates
  static constexpr size_t kCandBytes = static_cast<size_t>(kEpiWarps) * kRowsPerWarp * kCand * 8;
  static size_t list_bytes(int k) { return static_cast<size_t>(NC) * k * 8; }
  static size_t fixed_bytes(int k) {
    return 1024 /*alignment slack*/ + kZBytes + kRowBytes + list_bytes(k) + kCandBytes +
           kBarBytes;
  }
  static int stages(int k) {
    const long long room = kSmemLimit - static_cast<long long>(fixed_bytes(k));
    const long long s = room / kStageBytes;
    return static_cast<int>(s > kMaxStages ? kMaxStages : s);
  }
  static size_t smem_bytes(int k) {
    return fixed_bytes(k) + static_cast<size_t>(stages(k)) * kStageBytes;
  }
};

struct ProjArgs {
  const float* L;          // base logits of depth d, request 0
  long long l_req_stride;  // floats between two requests' rows
  int V, H, k, rows, rows_per_req, col0, n_stages;
  int tiled;               // 1: W_out in the tiled layout (PCTREE_HEAD_TILED)
  float* part_m;           // [rows][n_parts] per-CTA max
  float* part_s;           // [rows][n_parts] per-CTA sum of exp
  float* part_z;           // [rows][n_parts][k] per-CTA top-k logits, best first
  int32_t* part_t;         // [rows][n_parts][k] their tokens
  // [rows] per row: (tag << 32) | order key of the best k-th list entry of
  // any CTA; entries of earlier stages carry smaller tags and count as empty
  unsigned long long* gthr;
  unsigned tag;            // stage + 1
  int32_t* status;
};

// Order-preserving 32-bit key of a float (a larger float gives a larger
// unsigned key; no NaNs reach it) and its inverse.
__device__ __forceinline__ uint32_t float_key(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key_float(uint32_t key) {
  return __uint_as_float((key & 0x80000000u) ? (key & 0x7fffffffu) : ~key);
}

__device__ __forceinline__ void epi_barrier() { named_barrier(1, kEpiThreads); }


template <int NC>
__global__ void __launch_bounds__(kThreads, 1)
markov_fused_kernel(const __grid_constant__ CUtensorMap tmap_w,
                    const __grid_constant__ CUtensorMap tmap_x,
                    const __grid_constant__ ProjArgs a) {
  using C = FusedProj<NC>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* base = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int n_stages = a.n_stages;
  const int k = a.k;
  unsigned char* ring = base;
  float(*zs)[kBM] = reinterpret_cast<float(*)[kBM]>(ring + n_stages * C::kStageBytes);
  float* row_m = reinterpret_cast<float*>(reinterpret_cast<unsigned char*>(zs) + C::kZBytes);
  float* row_s = row_m + NC;
  float* thr_v = row_s + NC;                          // the list's k-th entry
  float* lv = thr_v + NC;                             // [NC][k]
  int* lt = reinterpret_cast<int*>(lv + NC * k);      // [NC][k]
  float* cbv = reinterpret_cast<float*>(lt + NC * k);  // [warp][row][kCand]
  int* cbt = reinterpret_cast<int*>(cbv + kEpiWarps * kRowsPerWarp * kCand);
  uint64_t* bars = reinterpret_cast<uint64_t*>(cbt + kEpiWarps * kRowsPerWarp * kCand);
  uint64_t* full = bars;                              // [kMaxStages]
  uint64_t* empty = bars + kMaxStages;                // [kMaxStages]
  uint64_t* acc_full = bars + 2 * kMaxStages;         // [kAccBufs]
  uint64_t* acc_empty = acc_full + 4;                 // [kAccBufs]
  uint64_t* drain = acc_empty + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
  int* stop_flag = abort_flag + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n_tiles = (a.V + kBM - 1) / kBM;
  const int n_k = (a.H + kBK - 1) / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < n_stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < C::kAccBufs; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kEpiWarps);   // one arrival per epilogue warp
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    *stop_flag = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tmap_w);
    tma_prefetch_desc(&tmap_x);
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_base = *tmem_slot;
  volatile int* abort_v = abort_flag;
  // the set-up above overlaps the previous kernel of the stream (the merge
  // that wrote this stage's parent rows); nothing below runs before it is
  // complete
  pdl_launch_dependents();
  pdl_wait();

  if (warp == 0) {
    // --------------------------------------------------------------- producer
    if (lane == 0) {
      const uint64_t stream_policy = l2_policy_evict_first();
      int stage = 0;
      uint32_t phase = 0;
      // ring slots holding a copy issued here, and the phase each was armed in
      uint32_t armed = 0, armed_phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
        for (int kc = 0; kc < n_k; ++kc) {
          if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, abort_v, kWaitLimitNs)) {
            ok = false;
            break;
          }
          unsigned char* a_dst = ring + stage * C::kStageBytes;
          int wx, wy;
          w_box(a.tiled, tile, kc, n_k, wx, wy);
          mbar_arrive_expect_tx(&full[stage], C::kStageBytes);
          tma_load_2d_hint(a_dst, &tmap_w, &full[stage], wx, wy, stream_policy);
          tma_load_2d(a_dst + C::kABytes, &tmap_x, &full[stage], kc * kBK, a.col0);
          armed |= 1u << stage;
          armed_phase = (armed_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == n_stages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        *abort_v = 1;
        set_status(a.status, PCTREE_ERR_TIMEOUT);
      }
      // every copy issued here must land before the CTA may exit
      volatile int never = 0;
      for (int s = 0; s < n_stages; ++s)
        if ((armed >> s) & 1u)
          mbar_wait_bounded(&full[s], (armed_phase >> s) & 1u, &never, kWaitLimitNs);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------- MMA issue
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, NC);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
        if (!mbar_wait_bounded(&acc_empty[acc], acc_phase ^ 1u, abort_v, kWaitLimitNs)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * NC);
        for (int kc = 0; kc < n_k; ++kc) {
          if (!mbar_wait_bounded(&full[stage], phase, abort_v, kWaitLimitNs)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t a_addr = smem_u32(ring + stage * C::kStageBytes);
          const uint32_t b_addr = a_addr + C::kABytes;
#pragma unroll
          for (int kk = 0; kk < kBK / kUmmaK; ++kk)
            tc_mma_bf16(d_tmem, desc_kmajor_sw128(a_addr + kk * kUmmaK * 2),
                        desc_kmajor_sw128(b_addr + kk * kUmmaK * 2), idesc,
                        (kc | kk) != 0 ? 1u : 0u);
          tc_commit(&empty[stage]);   // frees the ring slot once read
          if (++stage == n_stages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        tc_commit(&acc_full[acc]);    // accumulator ready for the epilogue
        if (++acc == C::kAccBufs) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
      if (!ok) {
        *abort_v = 1;
        set_status(a.status, PCTREE_ERR_TIMEOUT);
      }
      // every MMA issued here must be complete before TMEM is released
      tc_commit(drain);
      volatile int never = 0;
      mbar_wait_bounded(drain, 0, &never, kWaitLimitNs);
    }
  } else {
    // --------------------------------------------------------------- epilogue
    const int ew = warp - 2;                 // 0..7
    const int quad = warp & 3;               // TMEM lanes 32*quad .. +31
    const int half = ew >> 2;                // chunk columns 32*half .. +31
    const int tid = ew * 32 + lane;
    const int cols = min(NC, a.rows - a.col0);   // valid columns of this pass
    const int cols16 = (cols + 15) & ~15;
    // This warp's rows are c * 64 + 8 ew + i (chunk c, i < 8) in every
    // tile; each keeps a running (max, sum of exp) in shared memory (Eq. 2).
    constexpr int kChunks = (NC + kCC - 1) / kCC;
    for (int r = tid; r < NC; r += kEpiThreads) {
      row_m[r] = kNegInf;
      row_s[r] = 0.0f;
    }
    // The base logits a warp needs for one chunk: rows c * 64 + 8 ew + i,
    // this lane's four vocabulary entries of `tile`.  They are loaded one
    // chunk ahead (the next tile's first chunk during a tile's last), so the
    // loads' latency overlaps a chunk's work.
    auto load_l = [&](int tile, int c, float (&dst)[kRowsPerWarp][4]) {
#pragma unroll
      for (int i = 0; i < kRowsPerWarp; ++i) {
        const int rl = c * kCC + ew * kRowsPerWarp + i;
        const float* Lr = a.L + static_cast<long long>((a.col0 + (rl < cols ? rl : 0)) /
                                                       a.rows_per_req) * a.l_req_stride;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int v = tile * kBM + lane * 4 + e;
          dst[i][e] = (tile < n_tiles && rl < cols && v < a.V) ? __ldg(Lr + v) : 0.0f;
        }
      }
    };
    float lnx[kRowsPerWarp][4];
    load_l(blockIdx.x, 0, lnx);
    int acc = 0;
    uint32_t acc_phase = 0;
    bool bad = false;
    bool first = true;                       // this CTA's first tile
    for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
      // the lanes agree before the warp-collective TMEM loads; then one
      // decision for all eight warps, which meet at named barriers below
      const bool got = __all_sync(kFull, mbar_wait_bounded(&acc_full[acc], acc_phase,
                                                           abort_v, kWaitLimitNs));
      if (!got && lane == 0) {
        *abort_v = 1;
        set_status(a.status, PCTREE_ERR_TIMEOUT);
      }
      epi_barrier();
      if (tid == 0) *stop_flag = *abort_v;
      epi_barrier();
      if (*stop_flag) break;
      tc_fence_after_sync();
      const int v0 = tile * kBM;
      const int vb = v0 + lane * 4;          // this lane's 4 logits of a row
      const uint32_t t_lane = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                              static_cast<uint32_t>(acc * NC);
#pragma unroll 1
      for (int c = 0; c < kChunks; ++c) {
        const int c0 = c * kCC;
        if (c0 >= cols) break;
        // the shared threshold of this warp's row c0 + 8 ew + lane (lanes
        // 0..7), read past L1 now so that the load overlaps phase A
        float gl = kNegInf;
        {
          const int rl = c0 + ew * kRowsPerWarp + lane;
          if (!first && lane < kRowsPerWarp && rl < cols) {
            const unsigned long long w = __ldcg(a.gthr + a.col0 + rl);
            if (static_cast<unsigned>(w >> 32) == a.tag)
              gl = key_float(static_cast<uint32_t>(w));
          }
        }
        float lcur[kRowsPerWarp][4];
#pragma unroll
        for (int i = 0; i < kRowsPerWarp; ++i)
#pragma unroll
          for (int e = 0; e < 4; ++e) lcur[i][e] = lnx[i][e];
        if (c0 + kCC < cols)
          load_l(tile, c + 1, lnx);
        else
          load_l(tile + gridDim.x, 0, lnx);
        // A: 32 lanes x (up to) 32 columns of this warp's quadrant, transposed
        // into zs[column - c0][vocabulary row of the tile]
#pragma unroll
        for (int g = 0; g < 2; ++g) {
          const int cg = c0 + half * 32 + g * 16;
          if (cg < cols16) {
            uint32_t r[16];
            tmem_ld_32x32b_x16(t_lane + static_cast<uint32_t>(cg), r);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j) zs[cg - c0 + j][quad * 32 + lane] = __uint_as_float(r[j]);
          }
        }
        if (c0 + kCC >= cols) {
          // this warp's last TMEM read of the tile: hand the buffer back
          tc_fence_before_sync();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[acc]);
        }
        epi_barrier();
        // B: rows r0 .. r0 + 7 of the pass, processed together so that their
        // loads overlap (compile-time row indices keep every value in
        // registers)
        const int r0 = c0 + ew * kRowsPerWarp;       // pass-local rows
        const int nr = min(kRowsPerWarp, cols - r0);
        if (nr > 0) {
          float z[kRowsPerWarp][4];
#pragma unroll
          for (int i = 0; i < kRowsPerWarp; ++i) {
            const float4 acc4 = reinterpret_cast<const float4*>(zs[r0 - c0 + i])[lane];
            z[i][0] = acc4.x;
            z[i][1] = acc4.y;
            z[i][2] = acc4.z;
            z[i][3] = acc4.w;
          }
#pragma unroll
          for (int i = 0; i < kRowsPerWarp; ++i) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              if (i < nr && vb + e < a.V) {
                const float lval = lcur[i][e];
                // non-finite: a Markov bias that is not finite, or a NaN /
                // +inf base logit (-inf base logits are legal)
                bad |= !(fabsf(z[i][e]) < kPosInf) || !(lval < kPosInf);
                z[i][e] += lval;
              } else {
                z[i][e] = kNegInf;
              }
            }
          }
          // the tile's (max, sum of exp) of each row: eight warp reductions
          // side by side; lane i folds row i's pair into its running one
          float lm[kRowsPerWarp], es[kRowsPerWarp];
#pragma unroll
          for (int i = 0; i < kRowsPerWarp; ++i)
            lm[i] = fmaxf(fmaxf(z[i][0], z[i][1]), fmaxf(z[i][2], z[i][3]));
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
            for (int i = 0; i < kRowsPerWarp; ++i)
              lm[i] = fmaxf(lm[i], __shfl_xor_sync(kFull, lm[i], o));
          }
#pragma unroll
          for (int i = 0; i < kRowsPerWarp; ++i) {
            es[i] = 0.0f;
            if (lm[i] > kNegInf) {
              const float mb = lm[i] * kLog2e;
#pragma unroll
              for (int e = 0; e < 4; ++e) es[i] += ex2_approx(fmaf(z[i][e], kLog2e, -mb));
            }
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
            for (int i = 0; i < kRowsPerWarp; ++i)
              es[i] += __shfl_xor_sync(kFull, es[i], o);
          }
          {
            float my_m = kNegInf, my_s = 0.0f;
#pragma unroll
            for (int i = 0; i < kRowsPerWarp; ++i)
              if (lane == i) {
                my_m = lm[i];
                my_s = es[i];
              }
            if (lane < nr) {
              float m = row_m[r0 + lane], sm = row_s[r0 + lane];
              lse_merge(m, sm, my_m, my_s);
              row_m[r0 + lane] = m;
              row_s[r0 + lane] = sm;
            }
          }
          // the rows' logits go back to zs: the candidate compaction below
          // reads them there, so that z's registers are free for the lists
#pragma unroll
          for (int i = 0; i < kRowsPerWarp; ++i)
            reinterpret_cast<float4*>(zs[r0 - c0 + i])[lane] =
                make_float4(z[i][0], z[i][1], z[i][2], z[i][3]);
          // Top-k of each row over this CTA's tiles.  Bits 4i..4i+3 of `mk`
          // mark this lane's logits of row i that are candidates for the
          // row's list: at or above its k-th entry (in the first tile: those
          // left after seeding).
          uint32_t mk = 0;
          if (first) {
            // The list starts from the lanes' best logits, sorted by a warp
            // bitonic network; the eight rows go through it side by side
            // (every loop runs one operation for all rows before the next).
            float sv[kRowsPerWarp];
            int st[kRowsPerWarp], best[kRowsPerWarp];
#pragma unroll
            for (int i = 0; i < kRowsPerWarp; ++i) {
              sv[i] = z[i][0];
              st[i] = vb < a.V ? vb : 0x7fffffff;
              best[i] = 0;
#pragma unroll
              for (int e = 1; e < 4; ++e) {
                const int te = vb + e < a.V ? vb + e : 0x7fffffff;
                const bool bt = cand_better(z[i][e], te, sv[i], st[i]);
                sv[i] = bt ? z[i][e] : sv[i];
                st[i] = bt ? te : st[i];
                best[i] = bt ? e : best[i];
              }
              if (i >= nr) {
                sv[i] = kNegInf;
                st[i] = 0x7fffffff;
              }
            }
#pragma unroll
            for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
              for (int j = size >> 1; j > 0; j >>= 1) {
                float ov[kRowsPerWarp];
                int ot[kRowsPerWarp];
#pragma unroll
                for (int i = 0; i < kRowsPerWarp; ++i) ov[i] = __shfl_xor_sync(kFull, sv[i], j);
#pragma unroll
                for (int i = 0; i < kRowsPerWarp; ++i) ot[i] = __shfl_xor_sync(kFull, st[i], j);
                const bool take_best = ((lane & j) == 0) == ((lane & size) == 0);
#pragma unroll
                for (int i = 0; i < kRowsPerWarp; ++i) {
                  const bool b1 = cand_better(ov[i], ot[i], sv[i], st[i]);
                  const bool b2 = cand_better(sv[i], st[i], ov[i], ot[i]);
                  const bool sw = (take_best & b1) | (!take_best & b2);
                  sv[i] = sw ? ov[i] : sv[i];
                  st[i] = sw ? ot[i] : st[i];
                }
              }
            }
            float tv[kRowsPerWarp];
            int tt[kRowsPerWarp];
#pragma unroll
            for (int i = 0; i < kRowsPerWarp; ++i) tv[i] = __shfl_sync(kFull, sv[i], k - 1);
#pragma unroll
            for (int i = 0; i < kRowsPerWarp; ++i) tt[i] = __shfl_sync(kFull, st[i], k - 1);
#pragma unroll
            for (int i = 0; i < kRowsPerWarp; ++i) {
              if (i < nr) {
                const int rl = r0 + i;
                if (lane < k) {
                  lv[rl * k + lane] = sv[i];
                  lt[rl * k + lane] = st[i];
                }
                if (lane == k - 1) thr_v[rl] = sv[i];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const int te = vb + e < a.V ? vb + e : 0x7fffffff;
                  const bool m = (e != best[i]) & cand_better(z[i][e], te, tv[i], tt[i]);
                  mk |= static_cast<uint32_t>(m) << (4 * i + e);
                }
              }
            }
            __syncwarp();
          } else {
#pragma unroll
            for (int i = 0; i < kRowsPerWarp; ++i) {
              const float gi = __shfl_sync(kFull, gl, i);
              if (i < nr) {
                const float tv = fmaxf(thr_v[r0 + i], gi);
#pragma unroll
                for (int e = 0; e < 4; ++e)
                  if (z[i][e] >= tv && vb + e < a.V) mk |= 1u << (4 * i + e);
              }
            }
          }
          // lane i: row r0 + i's list changed in this chunk
          bool changed = first;
          if (__any_sync(kFull, mk != 0)) {
            // Candidates are few, so one lane per row inserts them into the
            // row's list in shared memory.  Each round compacts up to kCand
            // candidates per row (ballots, in (entry, lane) order) into this
            // warp's buffer; lane i then walks row i's candidates, each one
            // placed by an insertion step (exact (value desc, token asc)
            // order; what falls below the k-th drops out).
            float* cv_w = cbv + ew * kRowsPerWarp * kCand;
            int* ct_w = cbt + ew * kRowsPerWarp * kCand;
            const unsigned below = (1u << lane) - 1u;
            while (__any_sync(kFull, mk != 0)) {
              int n_mine = 0;
#pragma unroll
              for (int i = 0; i < kRowsPerWarp; ++i) {
                int base = 0;
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const bool m = (mk >> (4 * i + e)) & 1u;
                  const unsigned b = __ballot_sync(kFull, m);
                  const int slot = base + __popc(b & below);
                  if (m && slot < kCand) {
                    cv_w[i * kCand + slot] = zs[r0 - c0 + i][lane * 4 + e];
                    ct_w[i * kCand + slot] = vb + e;
                    mk &= ~(1u << (4 * i + e));
                  }
                  base += __popc(b);
                }
                if (lane == i) n_mine = base < kCand ? base : kCand;
              }
              changed |= n_mine > 0;
              __syncwarp();
              if (k <= kRegList) {
                // the row's list in registers, four lanes per row: lane
                // 4 i + q holds entries 4 q .. 4 q + 3 of row r0 + i
                // (entries >= k are sentinels).  A candidate goes through
                // every entry at once: each lane compares it with its four
                // entries, takes the entry shifted out of the previous
                // lane's segment, and selects.
                const int ri = lane >> 2, q = lane & 3;
                const int rl = r0 + ri;
                const int n_row = __shfl_sync(kFull, n_mine, ri);
                const int n_max = __reduce_max_sync(kFull, n_row);
                float rv[4];
                int rt[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                  const int e = 4 * q + j;
                  const bool live = ri < nr && e < k;
                  rv[j] = live ? lv[rl * k + e] : kNegInf;
                  rt[j] = live ? lt[rl * k + e] : 0x7fffffff;
                }
                for (int c = 0; c < n_max; ++c) {
                  const bool act = c < n_row;
                  const float v = act ? cv_w[ri * kCand + c] : kNegInf;
                  const int t = act ? ct_w[ri * kCand + c] : 0x7fffffff;
                  bool bt[4];
#pragma unroll
                  for (int j = 0; j < 4; ++j) bt[j] = act & cand_better(v, t, rv[j], rt[j]);
                  const float pv = __shfl_up_sync(kFull, rv[3], 1);
                  const int pt = __shfl_up_sync(kFull, rt[3], 1);
                  const bool pb = (__shfl_up_sync(kFull, static_cast<int>(bt[3]), 1) != 0) & (q != 0);
#pragma unroll
                  for (int j = 3; j > 0; --j) {
                    rv[j] = bt[j - 1] ? rv[j - 1] : (bt[j] ? v : rv[j]);
                    rt[j] = bt[j - 1] ? rt[j - 1] : (bt[j] ? t : rt[j]);
                  }
                  rv[0] = pb ? pv : (bt[0] ? v : rv[0]);
                  rt[0] = pb ? pt : (bt[0] ? t : rt[0]);
                }
                if (ri < nr && n_row > 0) {
#pragma unroll
                  for (int j = 0; j < 4; ++j) {
                    const int e = 4 * q + j;
                    if (e < k) {
                      lv[rl * k + e] = rv[j];
                      lt[rl * k + e] = rt[j];
                    }
                    if (e == k - 1) thr_v[rl] = rv[j];
                  }
                }
              } else if (lane < nr) {
                const int rl = r0 + lane;
                float* Lv = lv + rl * k;
                int* Lt = lt + rl * k;
                float kv = Lv[k - 1];
                int kt = Lt[k - 1];
                for (int c = 0; c < n_mine; ++c) {
                  const float v = cv_w[lane * kCand + c];
                  const int t = ct_w[lane * kCand + c];
                  if (!cand_better(v, t, kv, kt)) continue;
                  int j = k - 1;
                  while (j > 0) {
                    const float pv = Lv[j - 1];
                    const int pt = Lt[j - 1];
                    if (!cand_better(v, t, pv, pt)) break;
                    Lv[j] = pv;
                    Lt[j] = pt;
                    --j;
                  }
                  Lv[j] = v;
                  Lt[j] = t;
                  kv = Lv[k - 1];
                  kt = Lt[k - 1];
                }
                thr_v[rl] = kv;
              }
              __syncwarp();
            }
          }
          // publish the rows' k-th entries for the other CTAs
          __syncwarp();
          if (lane < nr && changed) {
            const float tv = thr_v[r0 + lane];
            if (tv > kNegInf)
              atomicMax(a.gthr + a.col0 + r0 + lane,
                        (static_cast<unsigned long long>(a.tag) << 32) | float_key(tv));
          }
        }
        epi_barrier();   // zs is rewritten by the next chunk
      }
      first = false;
      if (++acc == C::kAccBufs) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
    if (bad) set_status(a.status, PCTREE_ERR_NONFINITE);
    // this CTA's partial of every row of the pass
    epi_barrier();
    if (!*stop_flag) {
      const size_t n_parts = gridDim.x;
      for (int rl = ew; rl < cols; rl += kEpiWarps) {
        const size_t p = static_cast<size_t>(a.col0 + rl) * n_parts + blockIdx.x;
        if (lane == 0) {
          a.part_m[p] = row_m[rl];
          a.part_s[p] = row_s[rl];
        }
        if (lane < k) {
          a.part_z[p * k + lane] = first ? kNegInf : lv[rl * k + lane];
          a.part_t[p * k + lane] = first ? 0x7fffffff : lt[rl * k + lane];
        }
      }
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  if (warp == 1) tmem_dealloc(tmem_base, C::kTmemCols);
}

template <int NC>
cudaError_t launch_nc(const CUtensorMap* tmap_w, const CUtensorMap* tmap_x,
                      ProjArgs a, int num_sms, cudaStream_t stream) {
  using C = FusedProj<NC>;
  const int stages = C::stages(a.k);
  if (stages < 2) return cudaErrorInvalidValue;
  const size_t smem = C::smem_bytes(a.k);
  static SmemLimit limit;
  cudaError_t e = limit.ensure(reinterpret_cast<const void*>(markov_fused_kernel<NC>),
                               kSmemLimit);
  if (e != cudaSuccess) return e;
  a.n_stages = stages;
  const int grid = fused_proj_parts(a.V, num_sms);
  const int rows = a.rows;
  // programmatic dependent launch: a pass may be scheduled while the kernel
  // before it finishes (the kernel waits for it before touching memory)
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  for (int col0 = 0; col0 < rows; col0 += NC) {
    a.col0 = col0;
    e = cudaLaunchKernelEx(&cfg, markov_fused_kernel<NC>, *tmap_w, *tmap_x, a);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace

int fused_proj_parts(int V, int num_sms) {
  const int n_tiles = (V + kBM - 1) / kBM;
  const int g = n_tiles < num_sms ? n_tiles : num_sms;
  return g < kFusedMaxGrid ? g : kFusedMaxGrid;   // partial slots per row
}

cudaError_t launch_markov_fused(const CUtensorMap* tmap_w, const CUtensorMap* tmap_x,
                                const float* L, long long l_req_stride, int V,
                                int H, int k, int rows, int rows_per_req, int bn, int tiled,
                                int num_sms, float* part_m, float* part_s,
                                float* part_z, int32_t* part_t,
                                unsigned long long* gthr, unsigned tag,
                                int32_t* status, cudaStream_t stream) {
  ProjArgs a{};
  a.L = L;
  a.l_req_stride = l_req_stride;
  a.V = V;
  a.H = H;
  a.k = k;
  a.rows = rows;
  a.rows_per_req = rows_per_req;
  a.tiled = tiled;
  a.part_m = part_m;
  a.part_s = part_s;
  a.part_z = part_z;
  a.part_t = part_t;
  a.gthr = gthr;
  a.tag = tag;
  a.status = status;
  switch (bn) {
    case 16: return launch_nc<16>(tmap_w, tmap_x, a, num_sms, stream);
    case 32: return launch_nc<32>(tmap_w, tmap_x, a, num_sms, stream);
    case 64: return launch_nc<64>(tmap_w, tmap_x, a, num_sms, stream);
    case 128: return launch_nc<128>(tmap_w, tmap_x, a, num_sms, stream);
    case 256: return launch_nc<256>(tmap_w, tmap_x, a, num_sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace pct
