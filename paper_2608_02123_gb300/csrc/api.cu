// Host side of the PCTree C ABI (include/pctree.h): argument checks,
// workspace layout, TMA descriptors and the launch sequence of one drafting
// round (Algorithm 1): init, then per stage d = 0..B-1 the Markov projection
// (Eq. 3), the chunked log-softmax / top-k partials (Eq. 2) and the merge
// (Eq. 4, pool push, frontier); finally the budgeted selection and packing.
#include <cstdio>
#include <cstring>
#include <mutex>
#include <vector>

#include "pctree_common.cuh"

namespace pct {
namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned(const void* p, size_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

// Memory the kernels may read through `p`: device or managed memory, or
// page-locked host memory mapped into the device's address space at the same
// address (the kernels then read it over the host link, with no copy).
// Pageable host memory the driver does not know is refused, so that no
// kernel faults on it.
bool device_readable(const void* p) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    (void)cudaGetLastError();
    return false;
  }
  switch (at.type) {
    case cudaMemoryTypeDevice:
    case cudaMemoryTypeManaged:
      return true;
    case cudaMemoryTypeHost:
      return at.devicePointer == p;
    default:
      return false;
  }
}

pctree_status check_config(const pctree_config* c) {
  if (c == nullptr) return PCTREE_ERR_INVALID_ARG;
  if (c->V < 1 || c->H < 1 || c->B < 1 || c->k < 1 || c->N < 1 ||
      c->batch < 1)
    return PCTREE_ERR_INVALID_ARG;
  if (c->k > c->V) return PCTREE_ERR_INVALID_ARG;
  if (c->weight_dtype != PCTREE_F32 && c->weight_dtype != PCTREE_BF16)
    return PCTREE_ERR_INVALID_ARG;
  if (c->mode != PCTREE_MODE_PARENT && c->mode != PCTREE_MODE_SHARED)
    return PCTREE_ERR_INVALID_ARG;
  if (c->head_layout != PCTREE_HEAD_ROWMAJOR && c->head_layout != PCTREE_HEAD_TILED)
    return PCTREE_ERR_INVALID_ARG;
  if (c->head_layout == PCTREE_HEAD_TILED && c->weight_dtype != PCTREE_BF16)
    return PCTREE_ERR_INVALID_ARG;
  if (c->weight_dtype == PCTREE_BF16 && (c->H % 8) != 0)
    return PCTREE_ERR_INVALID_ARG;
  if (c->k > PCTREE_MAX_K || c->N > PCTREE_MAX_N) return PCTREE_ERR_UNSUPPORTED;
  if (static_cast<long long>(c->batch) * c->k > PCTREE_MAX_ROWS)
    return PCTREE_ERR_UNSUPPORTED;
  const long long P = 1 + c->k + static_cast<long long>(c->B - 1) * c->k * c->k;
  if (P > PCTREE_MAX_POOL) return PCTREE_ERR_UNSUPPORTED;
  if (c->V > (1 << 30) || c->H > (1 << 20)) return PCTREE_ERR_UNSUPPORTED;
  return PCTREE_OK;
}

Layout make_layout(const pctree_config& c) {
  Layout l{};
  l.rows_max = c.batch * (c.mode == PCTREE_MODE_SHARED ? 1 : c.k);
  l.rows_pad = static_cast<int>(align_up(l.rows_max, 16));
  l.bn = l.rows_pad <= 16 ? 16 : l.rows_pad <= 32 ? 32 : l.rows_pad <= 64 ? 64
         : l.rows_pad <= 128 ? 128 : 256;
  l.ldz = static_cast<int>(align_up(c.V, 64));
  l.n_chunks = (c.V + kChunk - 1) / kChunk;
  // bf16 heads: one partial per (row, projection CTA); f32 heads: one per
  // vocabulary chunk of the stage logits Z
  l.part_slots = c.weight_dtype == PCTREE_BF16 ? kFusedMaxGrid : l.n_chunks;
  l.P = 1 + c.k + (c.B - 1) * c.k * c.k;
  l.x_elem = c.weight_dtype == PCTREE_BF16 ? 2 : 4;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes, kAlign);
    return o;
  };
  const size_t rows = static_cast<size_t>(l.rows_max);
  l.off_x = take(static_cast<size_t>(l.rows_pad) * c.H * l.x_elem);
  // stage logits Z: only the f32 path writes them
  l.off_z = take(c.weight_dtype == PCTREE_BF16 ? 0 : rows * l.ldz * sizeof(float));
  l.off_pm = take(rows * l.part_slots * sizeof(float));
  l.off_ps = take(rows * l.part_slots * sizeof(float));
  l.off_pz = take(rows * l.part_slots * c.k * sizeof(float));
  l.off_pt = take(rows * l.part_slots * c.k * sizeof(int32_t));
  l.off_pool_tok = take(static_cast<size_t>(c.batch) * l.P * sizeof(int32_t));
  l.off_pool_par = take(static_cast<size_t>(c.batch) * l.P * sizeof(int32_t));
  l.off_pool_s = take(static_cast<size_t>(c.batch) * l.P * sizeof(float2));
  l.off_front = take(static_cast<size_t>(c.batch) * c.k * sizeof(int32_t));
  // stage tickets and release flags, then one flag per (CTA boundary,
  // TMEM lane quadrant) for the tiles two CTAs share
  l.sync_bytes = (2 * static_cast<size_t>(c.B) + 4 * kFusedMaxGrid) * sizeof(int);
  l.off_sync = take(l.sync_bytes);
  const size_t fparts = static_cast<size_t>(kFusedRows) * kFusedMaxGrid;
  l.off_fpm = take(fparts * sizeof(float));
  l.off_fps = take(fparts * sizeof(float));
  l.off_fcz = take(fparts * c.k * sizeof(float));
  l.off_fct = take(fparts * c.k * sizeof(int32_t));
  l.off_xtok = take(static_cast<size_t>(c.batch) * c.k * sizeof(int32_t));
  // partial accumulators of shared tiles, [stage parity][boundary][row][128]
  l.off_fxch = l.rows_max <= kFusedRows
                   ? take(2 * fparts * kFusedTileRows * sizeof(float))
                   : l.off_xtok;
  l.off_gthr = take(rows * sizeof(unsigned long long));
  l.total = off;
  return l;
}

}  // namespace

// --------------------------------------------------------------------------
// per-device facts and the driver's tensor-map encoder (shared with the
// other translation units through pctree_common.cuh)
// --------------------------------------------------------------------------

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t,
                                   void*, const cuuint64_t*, const cuuint64_t*,
                                   const cuuint32_t*, const cuuint32_t*,
                                   CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion,
                                   CUtensorMapFloatOOBfill);

std::mutex g_mu;
// Test hook (pctree_debug_stall_stage): a stage of the fused round whose
// release is withheld, and the bound of every wait of that kernel.
int g_stall_stage = -1;
unsigned long long g_wait_limit_ns = 1000000000ull;
EncodeTiledFn g_encode = nullptr;
int g_num_sms[64] = {0};

pctree_status device_facts(int* num_sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64)
    return PCTREE_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_num_sms[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) !=
        cudaSuccess)
      return PCTREE_ERR_CUDA;
    g_num_sms[dev] = n;
  }
  if (g_encode == nullptr) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                         cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || fn == nullptr)
      return PCTREE_ERR_CUDA;
    g_encode = reinterpret_cast<EncodeTiledFn>(fn);
  }
  *num_sms = g_num_sms[dev];
  return PCTREE_OK;
}

pctree_status encode_bf16_map_nd(CUtensorMap* map, const void* base, int rank,
                                 const uint64_t* dims,
                                 const uint64_t* strides_bytes,
                                 const uint32_t* box) {
  if (g_encode == nullptr || rank < 1 || rank > 5) return PCTREE_ERR_CUDA;
  cuuint64_t d[5], st[4];
  cuuint32_t b[5], e[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    b[i] = box[i];
    e[i] = 1;
    if (i + 1 < rank) st[i] = strides_bytes[i];
  }
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank,
                        const_cast<void*>(base), d, st, b, e,
                        CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? PCTREE_OK : PCTREE_ERR_INVALID_ARG;
}

namespace {

// 2-D bf16 tensor [rows][cols] (cols contiguous), box = box_rows x 64 with
// the 128-byte swizzle the MMA descriptors expect.
pctree_status encode_bf16_map(CUtensorMap* map, const void* base, int rows,
                              int cols, int box_rows);

// W_out's tensor map: [V][H] boxes of 128 x 64, or the tiled layout as a
// [n_tiles * n_k * 128][64] matrix whose 128 x 64 boxes are contiguous.
pctree_status encode_head_map(CUtensorMap* map, const void* head_out,
                              const pctree_config& c) {
  if (c.head_layout == PCTREE_HEAD_TILED) {
    const long long rows = static_cast<long long>((c.V + 127) / 128) *
                           ((c.H + 63) / 64) * 128;
    if (rows > (1ll << 31) - 1) return PCTREE_ERR_UNSUPPORTED;
    return encode_bf16_map(map, head_out, static_cast<int>(rows), 64, 128);
  }
  return encode_bf16_map(map, head_out, c.V, c.H, 128);
}
pctree_status encode_bf16_map(CUtensorMap* map, const void* base, int rows,
                              int cols, int box_rows) {
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols),
                        static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                        const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? PCTREE_OK : PCTREE_ERR_INVALID_ARG;
}

// --------------------------------------------------------------------------
// kernel timing
// --------------------------------------------------------------------------

constexpr int kMaxTimed = 8192;
struct Profiler {
  bool on = false;
  std::vector<cudaEvent_t> ev;  // 2 per launch
  int used = 0;
} g_prof;

void prof_record(int slot, cudaStream_t stream) {
  if (!g_prof.on) return;
  const int i = g_prof.used * 2 + slot;
  if (g_prof.used >= kMaxTimed) return;
  cudaEventRecord(g_prof.ev[i], stream);
  if (slot == 1) ++g_prof.used;
}

pctree_status cuda_status(cudaError_t e) {
  return e == cudaSuccess ? PCTREE_OK : PCTREE_ERR_CUDA;
}

// The fused round kernel covers bf16 heads with at most 16 Markov rows per
// stage; larger parent batches take the per-stage kernels.
int g_path = PCTREE_PATH_AUTO;

bool fused_path(const pctree_config& c) {
  return g_path == PCTREE_PATH_AUTO && c.weight_dtype == PCTREE_BF16 &&
         c.batch * c.k <= kFusedRows && c.k <= kFusedMaxK;
}

pctree_status draft_fused(const pctree_config& c, const Layout& lay,
                          const float* base_logits, const void* head_emb,
                          const void* head_out, const int32_t* root_token,
                          const pctree_tree& out, unsigned char* ws,
                          int num_sms, cudaStream_t stream) {
  CUtensorMap tmap_w, tmap_x;
  pctree_status st = encode_head_map(&tmap_w, head_out, c);
  if (st != PCTREE_OK) return st;
  st = encode_bf16_map(&tmap_x, ws + lay.off_x, kFusedRows, c.H, kFusedRows);
  if (st != PCTREE_OK) return st;
  const int n_tiles = (c.V + 127) / 128;
  int grid = num_sms < n_tiles ? num_sms : n_tiles;
  if (grid > kFusedMaxGrid) grid = kFusedMaxGrid;
  FusedArgs a{};
  a.L = base_logits;
  a.V = c.V;
  a.H = c.H;
  a.B = c.B;
  a.k = c.k;
  a.batch = c.batch;
  a.shared = c.mode == PCTREE_MODE_SHARED ? 1 : 0;
  a.tiled = c.head_layout == PCTREE_HEAD_TILED ? 1 : 0;
  a.P = lay.P;
  a.n_k = (c.H + 63) / 64;
  a.n_tiles = n_tiles;
  a.pool_tok = reinterpret_cast<int32_t*>(ws + lay.off_pool_tok);
  a.pool_par = reinterpret_cast<int32_t*>(ws + lay.off_pool_par);
  a.pool_s = reinterpret_cast<float2*>(ws + lay.off_pool_s);
  a.front = reinterpret_cast<int32_t*>(ws + lay.off_front);
  a.xtok = reinterpret_cast<int32_t*>(ws + lay.off_xtok);
  a.E_in = head_emb;
  a.X = ws + lay.off_x;
  int* sync = reinterpret_cast<int*>(ws + lay.off_sync);
  a.stage_cnt = sync;
  a.ready = sync + c.B;
  a.part_m = reinterpret_cast<float*>(ws + lay.off_fpm);
  a.part_s = reinterpret_cast<float*>(ws + lay.off_fps);
  a.cand_z = reinterpret_cast<float*>(ws + lay.off_fcz);
  a.cand_t = reinterpret_cast<int32_t*>(ws + lay.off_fct);
  a.xflag = sync + 2 * c.B;
  a.xch = reinterpret_cast<float*>(ws + lay.off_fxch);
  a.status = out.status;
  a.limit_ns = g_wait_limit_ns;
  a.stall_stage = g_stall_stage;
  if (cudaMemsetAsync(out.status, 0, sizeof(int32_t), stream) != cudaSuccess ||
      cudaMemsetAsync(sync, 0, lay.sync_bytes, stream) != cudaSuccess)
    return PCTREE_ERR_CUDA;
  st = cuda_status(launch_init(c, lay, root_token, head_emb, ws, out.status,
                               stream));
  if (st != PCTREE_OK) return st;
  prof_record(0, stream);
  NvtxRange range("round_fused (all stages)");
  const cudaError_t e = launch_round_fused(&tmap_w, &tmap_x, a, grid, stream);
  prof_record(1, stream);
  if (e != cudaSuccess) return PCTREE_ERR_CUDA;
  return cuda_status(launch_pack(c, lay, ws, out, stream));
}

}  // namespace
}  // namespace pct

using namespace pct;

extern "C" {

int32_t pctree_version(void) { return 102; }

const char* pctree_status_string(int32_t s) {
  switch (s) {
    case PCTREE_OK: return "ok";
    case PCTREE_ERR_INVALID_ARG: return "invalid argument";
    case PCTREE_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case PCTREE_ERR_CUDA: return "CUDA error";
    case PCTREE_ERR_TIMEOUT: return "device wait timed out";
    case PCTREE_ERR_NONFINITE: return "non-finite input or no finite logit";
    case PCTREE_ERR_UNSUPPORTED: return "shape outside compiled limits";
    default: return "unknown status";
  }
}

pctree_status pctree_check_config(const pctree_config* cfg) {
  return check_config(cfg);
}

int32_t pctree_pool_capacity(const pctree_config* cfg) {
  if (check_config(cfg) != PCTREE_OK) return 0;
  return 1 + cfg->k + (cfg->B - 1) * cfg->k * cfg->k;
}

size_t pctree_workspace_bytes(const pctree_config* cfg) {
  if (check_config(cfg) != PCTREE_OK) return 0;
  return make_layout(*cfg).total;
}

pctree_status pctree_draft(const pctree_config* cfg, const float* base_logits,
                           const void* head_emb, const void* head_out,
                           const int32_t* root_token, const pctree_tree* out,
                           void* workspace, size_t workspace_bytes,
                           void* stream_ptr) {
  NvtxRange range("pctree_draft");
  pctree_status st = check_config(cfg);
  if (st != PCTREE_OK) return st;
  const pctree_config c = *cfg;
  if (base_logits == nullptr || head_emb == nullptr || head_out == nullptr ||
      root_token == nullptr || out == nullptr)
    return PCTREE_ERR_INVALID_ARG;
  if (out->n_nodes == nullptr || out->tokens == nullptr ||
      out->parent == nullptr || out->depth == nullptr || out->logp == nullptr ||
      out->position_ids == nullptr || out->mask == nullptr ||
      out->retrieve == nullptr || out->n_leaves == nullptr ||
      out->status == nullptr)
    return PCTREE_ERR_INVALID_ARG;
  const int n_pool_ptrs = (out->pool_token != nullptr) +
                          (out->pool_parent != nullptr) +
                          (out->pool_logp != nullptr);
  if (n_pool_ptrs != 0 && n_pool_ptrs != 3) return PCTREE_ERR_INVALID_ARG;
  if (!aligned(head_emb, 16) || !aligned(head_out, 16) ||
      !aligned(base_logits, 4))
    return PCTREE_ERR_INVALID_ARG;
  const Layout lay = make_layout(c);
  if (workspace == nullptr || !aligned(workspace, kAlign) ||
      workspace_bytes < lay.total)
    return PCTREE_ERR_WORKSPACE;
  int num_sms = 0;
  st = device_facts(&num_sms);
  if (st != PCTREE_OK) return st;
  if (!device_readable(base_logits) || !device_readable(root_token))
    return PCTREE_ERR_INVALID_ARG;

  cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);
  unsigned char* ws = static_cast<unsigned char*>(workspace);
  if (fused_path(c)) return draft_fused(c, lay, base_logits, head_emb, head_out,
                                        root_token, *out, ws, num_sms, stream);
  CUtensorMap tmap_w, tmap_x;
  if (c.weight_dtype == PCTREE_BF16) {
    st = encode_head_map(&tmap_w, head_out, c);
    if (st != PCTREE_OK) return st;
    st = encode_bf16_map(&tmap_x, ws + lay.off_x, lay.rows_pad, c.H, lay.bn);
    if (st != PCTREE_OK) return st;
  }

  if (cudaMemsetAsync(out->status, 0, sizeof(int32_t), stream) != cudaSuccess)
    return PCTREE_ERR_CUDA;
  st = cuda_status(launch_init(c, lay, root_token, head_emb, ws, out->status,
                               stream));
  if (st != PCTREE_OK) return st;
  float* Z = reinterpret_cast<float*>(ws + lay.off_z);
  const long long l_req_stride = static_cast<long long>(c.B) * c.V;
  static const char* const kStageNames[] = {
      "stage 0",  "stage 1",  "stage 2",  "stage 3",  "stage 4",  "stage 5",
      "stage 6",  "stage 7",  "stage 8",  "stage 9",  "stage 10", "stage 11",
      "stage 12", "stage 13", "stage 14", "stage 15", "stage 16+"};
  for (int d = 0; d < c.B; ++d) {
    NvtxRange stage_range(kStageNames[d < 16 ? d : 16]);
    const int rpq = rows_per_request(c, d);  // b_d (Sec. 4.1), or 1
    const int rows = c.batch * rpq;
    const float* L_d = base_logits + static_cast<size_t>(d) * c.V;
    prof_record(0, stream);
    cudaError_t e;
    int n_parts;
    if (c.weight_dtype == PCTREE_BF16) {
      // projection, normaliser and top-k partials in one pass over W_out
      n_parts = fused_proj_parts(c.V, num_sms);
      e = launch_markov_fused(&tmap_w, &tmap_x, L_d, l_req_stride, c.V, c.H, c.k,
                              rows, rpq, lay.bn, c.head_layout == PCTREE_HEAD_TILED,
                              num_sms,
                              reinterpret_cast<float*>(ws + lay.off_pm),
                              reinterpret_cast<float*>(ws + lay.off_ps),
                              reinterpret_cast<float*>(ws + lay.off_pz),
                              reinterpret_cast<int32_t*>(ws + lay.off_pt),
                              reinterpret_cast<unsigned long long*>(ws + lay.off_gthr),
                              static_cast<unsigned>(d + 1), out->status, stream);
      prof_record(1, stream);
    } else {
      n_parts = lay.n_chunks;
      e = launch_markov_f32(static_cast<const float*>(head_out),
                            reinterpret_cast<const float*>(ws + lay.off_x), L_d,
                            l_req_stride, Z, lay.ldz, c.V, c.H, rows, rpq,
                            out->status, stream);
      prof_record(1, stream);
      if (e == cudaSuccess) e = launch_partials(lay, c.k, c.V, rows, ws, out->status, stream);
    }
    if (e != cudaSuccess) return PCTREE_ERR_CUDA;
    st = cuda_status(launch_merge(c, lay, d, n_parts, head_emb, ws, out->status, stream));
    if (st != PCTREE_OK) return st;
  }
  return cuda_status(launch_pack(c, lay, ws, *out, stream));
}

size_t pctree_packed_head_bytes(const pctree_config* cfg) {
  if (check_config(cfg) != PCTREE_OK || cfg->weight_dtype != PCTREE_BF16) return 0;
  return packed_head_bytes(cfg->V, cfg->H);
}

pctree_status pctree_pack_head(const pctree_config* cfg, const void* head_out,
                               void* packed, void* stream) {
  NvtxRange range("pctree_pack_head");
  pctree_status st = check_config(cfg);
  if (st != PCTREE_OK) return st;
  if (cfg->weight_dtype != PCTREE_BF16 || head_out == nullptr || packed == nullptr ||
      !aligned(head_out, 16) || !aligned(packed, 16))
    return PCTREE_ERR_INVALID_ARG;
  int num_sms = 0;
  st = device_facts(&num_sms);
  if (st != PCTREE_OK) return st;
  return cuda_status(launch_pack_head(head_out, packed, cfg->V, cfg->H, num_sms,
                                      static_cast<cudaStream_t>(stream)));
}

pctree_status pctree_accept(const pctree_config* cfg, const pctree_tree* tree,
                            const int32_t* target_tokens,
                            int32_t* accepted_idx, int32_t* accepted_len,
                            int32_t* bonus_token, void* stream_ptr) {
  NvtxRange range("pctree_accept");
  pctree_status st = check_config(cfg);
  if (st != PCTREE_OK) return st;
  if (tree == nullptr || tree->n_nodes == nullptr || tree->tokens == nullptr ||
      tree->parent == nullptr || target_tokens == nullptr ||
      accepted_idx == nullptr || accepted_len == nullptr ||
      bonus_token == nullptr)
    return PCTREE_ERR_INVALID_ARG;
  return cuda_status(launch_accept(*cfg, *tree, target_tokens, accepted_idx,
                                   accepted_len, bonus_token,
                                   static_cast<cudaStream_t>(stream_ptr)));
}

pctree_status pctree_debug_stall_stage(int32_t stage, int64_t wait_limit_ns) {
  if (stage < -1 || wait_limit_ns < 1000 || wait_limit_ns > 10000000000ll)
    return PCTREE_ERR_INVALID_ARG;
  g_stall_stage = stage;
  g_wait_limit_ns = static_cast<unsigned long long>(wait_limit_ns);
  return PCTREE_OK;
}

pctree_status pctree_set_path(int32_t path) {
  if (path != PCTREE_PATH_AUTO && path != PCTREE_PATH_STAGEWISE)
    return PCTREE_ERR_INVALID_ARG;
  g_path = path;
  return PCTREE_OK;
}

pctree_status pctree_profile_enable(int32_t on) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (on && g_prof.ev.empty()) {
    g_prof.ev.resize(2 * kMaxTimed);
    for (auto& e : g_prof.ev)
      if (cudaEventCreate(&e) != cudaSuccess) return PCTREE_ERR_CUDA;
  }
  g_prof.on = on != 0;
  g_prof.used = 0;
  return PCTREE_OK;
}

pctree_status pctree_profile_collect(int64_t* launches, double* total_ms) {
  if (launches == nullptr || total_ms == nullptr) return PCTREE_ERR_INVALID_ARG;
  double sum = 0.0;
  for (int i = 0; i < g_prof.used; ++i) {
    if (cudaEventSynchronize(g_prof.ev[2 * i + 1]) != cudaSuccess)
      return PCTREE_ERR_CUDA;
    float ms = 0.0f;
    if (cudaEventElapsedTime(&ms, g_prof.ev[2 * i], g_prof.ev[2 * i + 1]) !=
        cudaSuccess)
      return PCTREE_ERR_CUDA;
    sum += ms;
  }
  *launches = g_prof.used;
  *total_ms = sum;
  g_prof.used = 0;
  return PCTREE_OK;
}

}  // extern "C"
