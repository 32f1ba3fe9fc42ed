// Markov projection of one PCTree stage (Eq. 3) on GB300:
//
//   Z[row][v] = L_d[req(row)][v] + sum_h W_out[v][h] * X[row][h]
//
// where X[row] = E_in[parent token of row] (gathered by the previous stage)
// so that sum_h W_out[v][h] X[row][h] is the Markov head's bias for that
// parent.  The head matrix W_out (V x H, up to 1.5 GB) is streamed from HBM
// once per stage for every parent of every request, which makes this kernel
// the round's bandwidth bottleneck.
//
// bf16 path ("swap-AB"): the vocabulary is the MMA M dimension (128 rows per
// tile) and the stage's parent rows are the N dimension (16..256), so one
// W_out tile feeds every parent.  Persistent CTAs (one per SM) stream W_out
// tiles with TMA into a multi-stage shared-memory ring; one thread issues
// tcgen05.mma (bf16 x bf16 -> f32) into a double-buffered TMEM accumulator;
// four epilogue warps read it back with tcgen05.ld, add the base logits and
// store Z.  Warp roles:
//   warp 0      TMA producer
//   warp 1      TMEM allocator + MMA issuer
//   warps 2..5  epilogue (TMEM lane quadrant = warp % 4)
//
// f32 path: a plain CUDA-core kernel with float32 accumulation (tensor cores
// would round f32 inputs to tf32).
#include "pctree_common.cuh"
#include "sm103_ptx.cuh"

namespace pct {

namespace {

constexpr int kBM = 128;          // vocabulary rows per tile (MMA M)
constexpr int kBK = 64;           // K elements per ring stage (128 B of bf16)
constexpr int kUmmaK = 16;        // K per tcgen05.mma kind::f16
constexpr int kThreads = 192;
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // 1 s per bounded wait
constexpr int kLGroup = 16;       // requests whose base logits load together

template <int BN>
struct TcCfg {
  static constexpr int kABytes = kBM * kBK * 2;    // 16 KB
  static constexpr int kBBytes = BN * kBK * 2;     // 2..32 KB
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStages =
      (200 * 1024 / kStageBytes) > 8 ? 8 : (200 * 1024 / kStageBytes);
  static constexpr int kTmemCols =
      (2 * BN) <= 32 ? 32 : (2 * BN) <= 64 ? 64 : (2 * BN) <= 128 ? 128
                        : (2 * BN) <= 256 ? 256 : 512;
  static constexpr size_t kLBytes = kLGroup * kBM * sizeof(float);
  static constexpr size_t kSmemBytes =
      1024 /*alignment slack*/ + static_cast<size_t>(kStages) * kStageBytes +
      kLBytes + 256 /*barriers*/;
};

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
markov_tc_kernel(const __grid_constant__ CUtensorMap tmap_w,
                 const __grid_constant__ CUtensorMap tmap_x,
                 const float* __restrict__ L, long long l_req_stride,
                 float* __restrict__ Z, int ldz, int V, int H, int rows,
                 int rows_per_req, int col0, int32_t* status) {
  using C = TcCfg<BN>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* ring = smem;
  // base logits of up to kLGroup requests at each epilogue thread's
  // vocabulary entry ([request][row of tile]; each thread owns its column)
  float(*sl)[kBM] = reinterpret_cast<float(*)[kBM]>(ring + C::kStages * C::kStageBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring + C::kStages * C::kStageBytes +
                                               C::kLBytes);
  uint64_t* full = bars;                      // [kStages]
  uint64_t* empty = bars + C::kStages;        // [kStages]
  uint64_t* acc_full = bars + 2 * C::kStages; // [2]
  uint64_t* acc_empty = acc_full + 2;         // [2]
  uint64_t* drain = acc_empty + 2;            // [1]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n_tiles = (V + kBM - 1) / kBM;
  const int n_k = (H + kBK - 1) / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 4);  // one arrival per epilogue warp
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
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

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t stream_policy = l2_policy_evict_first();
      int stage = 0;
      uint32_t phase = 0;
      int armed[8];
      for (int s = 0; s < 8; ++s) armed[s] = -1;
      bool ok = true;
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
        for (int kc = 0; kc < n_k; ++kc) {
          if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, abort_v, kWaitLimitNs)) {
            ok = false;
            break;
          }
          unsigned char* a_dst = ring + stage * C::kStageBytes;
          unsigned char* b_dst = a_dst + C::kABytes;
          mbar_arrive_expect_tx(&full[stage], C::kStageBytes);
          tma_load_2d_hint(a_dst, &tmap_w, &full[stage], kc * kBK, tile * kBM,
                           stream_policy);
          tma_load_2d(b_dst, &tmap_x, &full[stage], kc * kBK, col0);
          armed[stage] = static_cast<int>(phase);
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        *abort_v = 1;
        set_status(status, PCTREE_ERR_TIMEOUT);
      }
      // Before the CTA may exit, every copy this thread issued must have
      // landed (a TMA write into freed shared memory would be unsafe).
      for (int s = 0; s < C::kStages; ++s) {
        if (armed[s] >= 0) {
          volatile int never = 0;
          mbar_wait_bounded(&full[s], static_cast<uint32_t>(armed[s]), &never,
                            kWaitLimitNs);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issue
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, BN);
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
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
        for (int kc = 0; kc < n_k; ++kc) {
          if (!mbar_wait_bounded(&full[stage], phase, abort_v, kWaitLimitNs)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t a_addr = smem_u32(ring + stage * C::kStageBytes);
          const uint32_t b_addr = a_addr + C::kABytes;
#pragma unroll
          for (int kk = 0; kk < kBK / kUmmaK; ++kk) {
            const uint64_t ad = desc_kmajor_sw128(a_addr + kk * kUmmaK * 2);
            const uint64_t bd = desc_kmajor_sw128(b_addr + kk * kUmmaK * 2);
            tc_mma_bf16(d_tmem, ad, bd, idesc, (kc | kk) != 0 ? 1u : 0u);
          }
          tc_commit(&empty[stage]);  // frees the ring slot once read
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        tc_commit(&acc_full[acc]);   // accumulator ready for the epilogue
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      if (!ok) {
        *abort_v = 1;
        set_status(status, PCTREE_ERR_TIMEOUT);
      }
      // wait for every MMA issued here before TMEM is released
      tc_commit(drain);
      volatile int never = 0;
      mbar_wait_bounded(drain, 0, &never, kWaitLimitNs);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quad = warp & 3;                 // TMEM lanes 32*quad .. +31
    const int r_in_tile = quad * 32 + lane;
    const int cols = min(BN, rows - col0);     // valid columns of this pass
    int acc = 0;
    uint32_t acc_phase = 0;
    bool bad = false;
    const int req_lo = col0 / rows_per_req;
    const int req_hi = (col0 + cols - 1) / rows_per_req;
    bool ok = true;
    for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
      const int v = tile * kBM + r_in_tile;
      const bool inb = v < V;
      const uint32_t t_row = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                             static_cast<uint32_t>(acc * BN);
      for (int g0 = req_lo; g0 <= req_hi; g0 += kLGroup) {
        // the group's base logits, as independent loads issued together
        // (for the first group: before the accumulator wait)
        float lv[kLGroup];
#pragma unroll
        for (int q = 0; q < kLGroup; ++q)
          lv[q] = inb && g0 + q <= req_hi
                      ? __ldg(L + static_cast<long long>(g0 + q) * l_req_stride + v)
                      : 0.0f;
        if (g0 == req_lo) {
          // the lanes agree before the warp-collective TMEM loads
          if (!__all_sync(0xffffffffu, mbar_wait_bounded(&acc_full[acc], acc_phase,
                                                         abort_v, kWaitLimitNs))) {
            *abort_v = 1;
            set_status(status, PCTREE_ERR_TIMEOUT);
            ok = false;
            break;
          }
          tc_fence_after_sync();
        }
#pragma unroll
        for (int q = 0; q < kLGroup; ++q) sl[q][r_in_tile] = lv[q];
        // pass-relative columns of the group's requests
        const int c_lo = max(col0, g0 * rows_per_req) - col0;
        const int c_hi = min(col0 + cols, (g0 + kLGroup) * rows_per_req) - col0;
        int q = (col0 + c_lo) / rows_per_req - g0;      // request of column c_lo
        int next = (g0 + q + 1) * rows_per_req - col0;  // its first column after
        for (int c0 = c_lo & ~15; c0 < c_hi; c0 += 16) {
          uint32_t r[16];
          tmem_ld_32x32b_x16(t_row + c0, r);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int c = c0 + j;
            if (c >= c_lo && c < c_hi) {
              if (c == next) {
                ++q;
                next += rows_per_req;
              }
              if (inb) {
                const float lval = sl[q][r_in_tile];
                const float z = lval + __uint_as_float(r[j]);
                bad |= isnan(z) || (isinf(z) && !(isinf(lval) && lval < 0.0f));
                Z[static_cast<size_t>(col0 + c) * ldz + v] = z;
              }
            }
          }
        }
      }
      if (!ok) break;
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[acc]);
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
    if (bad) set_status(status, PCTREE_ERR_NONFINITE);
  }

  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  if (warp == 1) tmem_dealloc(tmem_base, C::kTmemCols);
}

template <int BN>
cudaError_t launch_tc(const CUtensorMap* tmap_w, const CUtensorMap* tmap_x,
                      const float* L, long long l_req_stride, float* Z,
                      int ldz, int V, int H, int rows, int rows_per_req,
                      int num_sms, int32_t* status, cudaStream_t stream) {
  using C = TcCfg<BN>;
  static SmemLimit limit;
  {
    cudaError_t e = limit.ensure(reinterpret_cast<const void*>(markov_tc_kernel<BN>),
                                 C::kSmemBytes);
    if (e != cudaSuccess) return e;
  }
  const int n_tiles = (V + kBM - 1) / kBM;
  const int grid = n_tiles < num_sms ? n_tiles : num_sms;
  for (int col0 = 0; col0 < rows; col0 += BN) {
    markov_tc_kernel<BN><<<grid, kThreads, C::kSmemBytes, stream>>>(
        *tmap_w, *tmap_x, L, l_req_stride, Z, ldz, V, H, rows, rows_per_req,
        col0, status);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

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

cudaError_t launch_markov_bf16(const CUtensorMap* tmap_w,
                               const CUtensorMap* tmap_x, const float* L,
                               long long l_req_stride, float* Z, int ldz,
                               int V, int H, int rows, int rows_per_req,
                               int bn, int num_sms, int32_t* status,
                               cudaStream_t stream) {
  switch (bn) {
    case 16:
      return launch_tc<16>(tmap_w, tmap_x, L, l_req_stride, Z, ldz, V, H, rows,
                           rows_per_req, num_sms, status, stream);
    case 32:
      return launch_tc<32>(tmap_w, tmap_x, L, l_req_stride, Z, ldz, V, H, rows,
                           rows_per_req, num_sms, status, stream);
    case 64:
      return launch_tc<64>(tmap_w, tmap_x, L, l_req_stride, Z, ldz, V, H, rows,
                           rows_per_req, num_sms, status, stream);
    case 128:
      return launch_tc<128>(tmap_w, tmap_x, L, l_req_stride, Z, ldz, V, H,
                            rows, rows_per_req, num_sms, status, stream);
    case 256:
      return launch_tc<256>(tmap_w, tmap_x, L, l_req_stride, Z, ldz, V, H,
                            rows, rows_per_req, num_sms, status, stream);
    default:
      return cudaErrorInvalidValue;
  }
}

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
