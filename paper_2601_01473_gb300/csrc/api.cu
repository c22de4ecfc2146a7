// api.cu -- the C ABI of libagnes.so (declared in include/agnes.h).
//
// Orchestrates one hyperbatch (Algorithm 1, Sec. 3.5) on the caller's stream:
//   bucket the targets by (tile, minibatch)                   [sample.cu]
//   for each hop: count min(deg, k) per frontier entry, scan to indptr,
//                 sample in bucket order                      [sample.cu, scan.cu]
//                 bucket the samples, dedup + relabel, carry the bucket
//                                                             [dedup.cu]
//   gather the final bucket's rows block by block             [gather.cu]
//   count the blocks touched (the paper's block-wise I/Os)   [gather.cu]
// Everything is sized for the worst case up front (per-minibatch capacities
// cap_h = min(N, B * prod(1 + k))), so no kernel's launch waits on a count
// from the device and the host synchronises only when a view is fetched.
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <new>
#include <vector>

#include "../../include/agnes.h"
#include "common.cuh"
#include "internal.h"

using namespace agnes;

namespace {

constexpr int kMaxPhases = 2 + 3 * AGNES_MAX_HOPS;
constexpr int kEventRing = 64;  // prepares whose phase times stay readable
// Streaming of host-resident features: a ring of staging slots in HBM, each
// holding a batch of up to kStreamBatchBlocks touched feature blocks.
constexpr int kStreamSlots = 4;
constexpr int kStreamBatchBlocks = 64;
// In-place topology reads with a topology cache: hyperbatches between re-picks
// of the cached block runs.
constexpr int64_t kTopoRepickEvery = 8;

struct Workspace {
  int32_t H = 0, B = 0, K = 0;
  int32_t fan[AGNES_MAX_HOPS] = {0};
  int64_t cap[AGNES_MAX_HOPS + 1] = {0};
  int64_t capK = 0, ecap_max = 0, cap_prev_max = 0;
  bool valid = false;

  int32_t* nodes = nullptr;
  int32_t* fb_id[2] = {nullptr, nullptr};
  int32_t* fb_pos[2] = {nullptr, nullptr};
  int32_t* fcell_off[2] = {nullptr, nullptr};
  int32_t* fcnt = nullptr;
  int32_t* scnt = nullptr;
  int32_t* soff = nullptr;
  int32_t* nfcnt = nullptr;
  int32_t* newcnt = nullptr;
  int32_t* newbase = nullptr;
  int32_t* nsz = nullptr;   // (K+1) x H: |dst_h| (h < K), |src_{K-1}| (h = K)
  int32_t* srcsz = nullptr; // K x H: |src_h|
  int32_t* noutbase = nullptr;  // T*H: sampled frontier: per-minibatch scan of next-frontier counts
  int32_t* ecnt = nullptr;  // K x H
  int64_t* indptr[AGNES_MAX_HOPS] = {nullptr};
  int32_t* col[AGNES_MAX_HOPS] = {nullptr};
  int32_t* nbr = nullptr;
  int32_t* scell = nullptr;
  int32_t* srank = nullptr;
  int2* sb = nullptr;
  int2* tmp = nullptr;
  int32_t* big_list = nullptr;
  int32_t* big_n = nullptr;
  int32_t* tmp_id = nullptr;
  int32_t* tmp_pos = nullptr;
  int32_t* cnt = nullptr;
  void* feats_out = nullptr;
  uint8_t* adj_flags = nullptr;
  uint8_t* feat_flags = nullptr;
  int64_t* stats = nullptr;  // K+1
  int64_t* scan_scratch = nullptr;
  int32_t* status = nullptr;
  unsigned long long* distinct = nullptr;
  uint64_t* key = nullptr;  // sampling key {seed, first minibatch id}

  // pinned host readback: [status][nsz (K+1)H][ecnt KH][srcsz KH] then int64 stats (K+1)
  void* h_back = nullptr;
  size_t h_back_bytes = 0;
};

}  // namespace

struct agnes_ctx {
  int device = 0;
  int num_sms = 0;
  cudaStream_t load_stream = nullptr;

  int64_t N = 0, E = 0;
  int offsets_bits = 64;
  void* offsets = nullptr;
  int32_t* indices = nullptr;
  void* features = nullptr;
  bool own_offsets = false, own_indices = false, own_features = false;
  int32_t feat_dtype = 0;
  int64_t feat_dim = 0, row_bytes = 0;
  int32_t features_on_host = 0;
  void* scratch = nullptr;  // ctx_scratch
  size_t scratch_bytes = 0;
  void* pinned = nullptr;   // ctx_pinned
  size_t pinned_bytes = 0;
  int32_t feature_io = AGNES_FEATURE_IO_BLOCKS;
  int32_t frontier_mode = AGNES_FRONTIER_SRC;
  const char* features_dev = nullptr;  // device view of host-resident features
  int64_t adj_block_bytes = 0, feat_block_bytes = 0;
  BlockTables bt;

  Workspace ws;
  bool prepared = false;
  bool synced = false;
  int cur = 0;  // which frontier buffer holds the final bucket
  cudaEvent_t done = nullptr;

  bool profiling = false;
  int64_t n_prepared = 0;                  // prepares issued so far
  int n_phases[kEventRing] = {0};          // per ring slot; 0 = not profiled
  cudaEvent_t ev[kEventRing][kMaxPhases + 1] = {{nullptr}};
  bool ev_created = false;
  uint64_t ws_gen = 0;  // bumped whenever the workspace is reallocated

  // The resident path's launch sequence, captured once per hyperbatch shape
  // and replayed as one CUDA graph launch (agnes_set_launch_mode).
  struct LaunchGraph {
    int32_t mode = AGNES_LAUNCH_GRAPH_PDL;
    cudaStream_t cap = nullptr;  // private stream the sequence is captured on
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    // what the capture depends on
    int32_t H = 0, B = 0, K = 0, fan[AGNES_MAX_HOPS] = {0}, frontier_mode = 0, built_mode = 0;
    bool profiling = false;
    uint64_t ws_gen = 0;
    // phase-event nodes, re-pointed at each launch's ring slot
    cudaGraphNode_t phase_node[kMaxPhases + 1] = {nullptr};
    int n_marks = 0;
    int64_t captures = 0, launches = 0, programmatic_edges = 0;
  } lg;

  // streaming of host-resident features (features_on_host)
  cudaStream_t copy_stream = nullptr;
  char* slots = nullptr;
  int64_t slot_bytes = 0;
  cudaEvent_t slot_copied[kStreamSlots] = {nullptr};
  cudaEvent_t slot_free[kStreamSlots] = {nullptr};
  bool slot_used[kStreamSlots] = {false};
  int32_t* d_counts = nullptr;   // requests per feature block (this hyperbatch)
  int32_t* h_counts = nullptr;   // pinned copy
  int32_t* h_touched = nullptr;  // pinned, touched feature blocks of the last hyperbatch
  int32_t* d_touched = nullptr;
  unsigned long long* h_src = nullptr;  // pinned: device address of each touched block's copy
  unsigned long long* d_src = nullptr;
  int32_t* h_job_blk = nullptr;         // pinned: blocks to load this hyperbatch ...
  int32_t* d_job_blk = nullptr;
  unsigned long long* h_job_dst = nullptr;  // ... and where to
  unsigned long long* d_job_dst = nullptr;
  unsigned long long* h_addr = nullptr;  // row mode: current address of every feature block
  unsigned long long* d_addr = nullptr;
  // row mode: requested-id bitmaps per tile, their word prefixes and counts,
  // the scan of the counts, the staging rows, and the rows read from host
  uint32_t* rm_bitmap = nullptr;
  uint16_t* rm_wpref = nullptr;
  int32_t* rm_dcnt = nullptr;
  int32_t* rm_doff = nullptr;
  char* rm_staging = nullptr;
  int64_t rm_staging_rows = 0;
  unsigned long long* d_host_rows = nullptr;
  int64_t* h_rm = nullptr;  // pinned: [0] distinct rows, [1] rows read from host memory
  int64_t cache_load_bytes = 0;
  cudaEvent_t gather_start = nullptr;
  // feature cache C_f (Sec. 3.4 (2)): blocks whose cumulative request count
  // reaches the threshold, hottest first, up to fcache_slots blocks
  int64_t fcache_slots = 0, fcache_threshold = 0;
  char* fcache = nullptr;
  std::vector<int64_t> acc;          // cumulative requests per feature block
  std::vector<int32_t> cslot_of;     // block -> cache slot, -1 if not admitted
  std::vector<int32_t> cblock_of;    // cache slot -> block, -1 if free
  std::vector<uint8_t> cresident;    // cache slot holds its block's rows
  int64_t fcache_hits = 0, fcache_loads = 0;
  std::vector<int32_t> fblock_first_tile;
  int64_t streamed_bytes = 0, streamed_blocks = 0;

  // topology in pinned host memory, HBM graph buffer with LRU + pinning
  struct Topo {
    bool on = false;
    const int32_t* host_indices = nullptr;
    const int32_t* dev_view = nullptr;  // device address of host_indices
    int64_t slots = 0, epb = 0;
    int2* d_jobs = nullptr;             // per wave: (block, slot) copies for the loader
    int2* h_jobs = nullptr;             // pinned staging of the jobs
    int32_t jobs_cap = 0;
    int32_t* gbuf = nullptr;
    int32_t* d_slot = nullptr;          // n_blocks: slot of each physical block, -1 if absent
    int32_t* h_slot_stage = nullptr;    // pinned staging for uploads of the slot table
    std::vector<int32_t> slot_of;       // host: block -> slot
    std::vector<int32_t> block_of;      // slot -> block or -1
    std::vector<int32_t> prev, next;    // LRU list over slots (head = least recent)
    int32_t head = -1, tail = -1;
    std::vector<uint32_t> pinned;       // slot -> wave it is pinned for (0: never)
    uint32_t wave = 2;                  // waves count from 3, so 0 is always evictable
    std::vector<int64_t> e0, e1;        // block edge ranges
    std::vector<int32_t> start_block;   // n_starts + 1 (sentinel n_blocks)
    std::vector<int32_t> run_first_tile;
    uint8_t* d_need = nullptr;
    uint8_t* h_need = nullptr;
    cudaStream_t copy = nullptr;
    cudaEvent_t uploaded = nullptr, wave_done[2] = {nullptr, nullptr};
    bool uploaded_used = false;
    int64_t loaded_blocks = 0, loaded_bytes = 0, hits = 0, waves = 0;
    uint64_t sweeps = 0;  // hops sampled so far (sets the sweep direction)
    // in-place reads (AGNES_TOPOLOGY_IO_ROWS) with a topology cache: gbuf holds
    // the most requested block runs, the sampler reads the rest in place
    bool cache = false;
    unsigned long long* d_acc = nullptr;   // n_starts: frontier entries per run since load
    unsigned long long* h_acc = nullptr;   // pinned read-back of d_acc (at re-picks)
    unsigned long long* d_cached = nullptr;  // frontier entries on cached blocks since load
    unsigned long long* h_cached = nullptr;  // pinned, read back after every hyperbatch
    std::vector<int32_t> run_of;        // n_blocks: block run of each physical block
  } topo;

  char err[512] = {0};
};

static thread_local char g_err[512];

static void set_err(agnes_ctx* ctx, const char* fmt, ...) {
  char* dst = ctx ? ctx->err : g_err;
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(dst, 512, fmt, ap);
  va_end(ap);
  if (ctx) snprintf(g_err, sizeof(g_err), "%s", ctx->err);
}

void ctx_graph_view(const agnes_ctx* ctx, agnes::GraphView* out) {
  out->device = ctx->device;
  out->num_sms = ctx->num_sms;
  out->offsets = ctx->offsets;
  out->offsets_bits = ctx->offsets_bits;
  out->N = ctx->N;
}

cudaError_t ctx_scratch(agnes_ctx* ctx, size_t bytes, void** out) {
  if (ctx->scratch_bytes < bytes) {
    cudaFree(ctx->scratch);
    ctx->scratch = nullptr;
    ctx->scratch_bytes = 0;
    const cudaError_t e = cudaMalloc(&ctx->scratch, bytes);
    if (e != cudaSuccess) return e;
    ctx->scratch_bytes = bytes;
  }
  *out = ctx->scratch;
  return cudaSuccess;
}

cudaError_t ctx_pinned(agnes_ctx* ctx, size_t bytes, void** out) {
  if (ctx->pinned_bytes < bytes) {
    if (ctx->pinned) cudaFreeHost(ctx->pinned);
    ctx->pinned = nullptr;
    ctx->pinned_bytes = 0;
    const cudaError_t e = cudaMallocHost(&ctx->pinned, bytes);
    if (e != cudaSuccess) return e;
    ctx->pinned_bytes = bytes;
  }
  *out = ctx->pinned;
  return cudaSuccess;
}

void ctx_set_error(agnes_ctx* ctx, const char* fmt, ...) {
  char* dst = ctx ? ctx->err : g_err;
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(dst, 512, fmt, ap);
  va_end(ap);
  if (ctx) snprintf(g_err, sizeof(g_err), "%s", ctx->err);
}

#define CK(ctx, call)                                                            \
  do {                                                                           \
    cudaError_t e_ = (call);                                                     \
    if (e_ != cudaSuccess) {                                                     \
      set_err(ctx, "%s failed: %s", #call, cudaGetErrorString(e_));              \
      return e_ == cudaErrorMemoryAllocation ? AGNES_ENOMEM : AGNES_ECUDA;       \
    }                                                                            \
  } while (0)

static bool is_device_ptr(const void* p) {
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged;
}

static bool is_pinned_host_ptr(const void* p) {
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return attr.type == cudaMemoryTypeHost;
}

namespace agnes {
namespace {
__global__ void fill_i32_kernel(int32_t* p, int64_t n, int32_t v) {
  grid_dep_wait();
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    p[i] = v;
}
}  // namespace
}  // namespace agnes

static void free_workspace(Workspace* w) {
  cudaFree(w->nodes);
  for (int b = 0; b < 2; ++b) {
    cudaFree(w->fb_id[b]);
    cudaFree(w->fb_pos[b]);
    cudaFree(w->fcell_off[b]);
  }
  cudaFree(w->fcnt);
  cudaFree(w->scnt);
  cudaFree(w->soff);
  cudaFree(w->nfcnt);
  cudaFree(w->newcnt);
  cudaFree(w->newbase);
  cudaFree(w->nsz);
  cudaFree(w->srcsz);
  cudaFree(w->noutbase);
  cudaFree(w->ecnt);
  for (int h = 0; h < AGNES_MAX_HOPS; ++h) {
    cudaFree(w->indptr[h]);
    cudaFree(w->col[h]);
  }
  cudaFree(w->nbr);
  cudaFree(w->scell);
  cudaFree(w->srank);
  cudaFree(w->sb);
  cudaFree(w->tmp);
  cudaFree(w->big_list);
  cudaFree(w->big_n);
  cudaFree(w->tmp_id);
  cudaFree(w->tmp_pos);
  cudaFree(w->cnt);
  cudaFree(w->feats_out);
  cudaFree(w->adj_flags);
  cudaFree(w->feat_flags);
  cudaFree(w->stats);
  cudaFree(w->scan_scratch);
  cudaFree(w->status);
  cudaFree(w->distinct);
  cudaFree(w->key);
  if (w->h_back) cudaFreeHost(w->h_back);
  *w = Workspace();
}

template <typename T>
static cudaError_t dalloc(T** p, int64_t n) {
  return cudaMalloc((void**)p, sizeof(T) * (size_t)(n > 0 ? n : 1));
}

static agnes_status ensure_workspace(agnes_ctx* ctx, int32_t H, int32_t B, const int32_t* fan,
                                     int32_t K, const int64_t* cap) {
  Workspace& w = ctx->ws;
  bool same = w.valid && w.H == H && w.B == B && w.K == K;
  for (int h = 0; same && h < K; ++h) same = w.fan[h] == fan[h];
  if (same) return AGNES_OK;
  cudaDeviceSynchronize();
  free_workspace(&w);
  ctx->ws_gen += 1;  // launch sequences captured over the old buffers are stale
  w.H = H;
  w.B = B;
  w.K = K;
  for (int h = 0; h < K; ++h) w.fan[h] = fan[h];
  for (int h = 0; h <= K; ++h) w.cap[h] = cap[h];
  w.capK = cap[K];
  w.ecap_max = 0;
  w.cap_prev_max = 0;
  for (int h = 0; h < K; ++h) {
    const int64_t e = cap[h] * fan[h];
    if (e > w.ecap_max) w.ecap_max = e;
    if (cap[h] > w.cap_prev_max) w.cap_prev_max = cap[h];
  }
  const int64_t T = ctx->bt.T;
  const int64_t cells = T * H;
  const int64_t rows = (int64_t)H * w.capK;
  const int64_t edges = (int64_t)H * w.ecap_max;
  const int64_t nb = ctx->bt.n_blocks;
  const int64_t nfb = ctx->bt.n_feat_blocks;
  int64_t scratch = scan_scratch_elems(1, cells);
  const int64_t s2 = scan_scratch_elems(1, ctx->N);
  const int64_t s3 = scan_scratch_elems(H, w.cap_prev_max);
  const int64_t s4 = col_scan_scratch_elems(T, H);
  if (s2 > scratch) scratch = s2;
  if (s3 > scratch) scratch = s3;
  if (s4 > scratch) scratch = s4;

#define WA(p, n)                                                                             \
  do {                                                                                       \
    if (dalloc(&(p), (n)) != cudaSuccess) {                                                  \
      cudaGetLastError();                                                                    \
      free_workspace(&w);                                                                    \
      set_err(ctx, "out of device memory allocating %s (%lld elements)", #p, (long long)(n)); \
      return AGNES_ENOMEM;                                                                   \
    }                                                                                        \
  } while (0)

  WA(w.nodes, rows);
  for (int b = 0; b < 2; ++b) {
    WA(w.fb_id[b], rows);
    WA(w.fb_pos[b], rows);
    WA(w.fcell_off[b], cells + 1);
  }
  WA(w.fcnt, cells);
  WA(w.scnt, cells);
  WA(w.soff, cells + 1);
  WA(w.nfcnt, cells);
  WA(w.newcnt, cells);
  WA(w.newbase, cells);
  WA(w.nsz, (int64_t)(K + 1) * H);
  WA(w.srcsz, (int64_t)K * H);
  WA(w.noutbase, cells);
  WA(w.ecnt, (int64_t)K * H);
  for (int h = 0; h < K; ++h) {
    WA(w.indptr[h], (int64_t)H * (cap[h] + 1));
    WA(w.col[h], (int64_t)H * cap[h] * fan[h]);
  }
  WA(w.nbr, edges);
  WA(w.scell, edges);
  WA(w.srank, edges);
  WA(w.sb, edges);
  WA(w.tmp, rows + edges);
  WA(w.big_list, (rows + edges) / (kDedupSmallMax + 1) + 1);
  WA(w.big_n, 1);
  WA(w.tmp_id, (int64_t)H * B);
  WA(w.tmp_pos, (int64_t)H * B);
  WA(w.cnt, (int64_t)H * w.cap_prev_max);
  {
    uint8_t* f = nullptr;
    WA(f, rows * ctx->row_bytes);
    w.feats_out = f;
  }
  WA(w.adj_flags, (int64_t)K * nb);
  WA(w.feat_flags, nfb);
  WA(w.stats, K + 1);
  WA(w.scan_scratch, scratch);
  WA(w.status, 1);
  WA(w.distinct, 1);
  WA(w.key, 2);
#undef WA
  w.h_back_bytes = sizeof(int32_t) * (1 + (size_t)(K + 1) * H + 2 * (size_t)K * H + 1) +
                   sizeof(int64_t) * (K + 2);
  if (cudaMallocHost(&w.h_back, w.h_back_bytes) != cudaSuccess) {
    cudaGetLastError();
    w.h_back = nullptr;
    free_workspace(&w);
    set_err(ctx, "out of pinned host memory");
    return AGNES_ENOMEM;
  }
  if (cudaMemset(w.scan_scratch, 0, sizeof(int64_t) * scratch) != cudaSuccess ||
      cudaMemset(w.fcnt, 0, sizeof(int32_t) * cells) != cudaSuccess ||
      cudaMemset(w.scnt, 0, sizeof(int32_t) * cells) != cudaSuccess) {
    free_workspace(&w);
    set_err(ctx, "cudaMemset failed");
    return AGNES_ECUDA;
  }
  w.valid = true;
  return AGNES_OK;
}

// Host view of the readback buffer.
struct Back {
  int32_t* status;
  int32_t* nsz;
  int32_t* ecnt;
  int32_t* srcsz;
  int64_t* stats;
};

static Back back_of(Workspace& w) {
  Back b;
  int32_t* p = (int32_t*)w.h_back;
  b.status = p;
  b.nsz = p + 1;
  b.ecnt = b.nsz + (size_t)(w.K + 1) * w.H;
  b.srcsz = b.ecnt + (size_t)w.K * w.H;
  size_t off32 = 1 + (size_t)(w.K + 1) * w.H + 2 * (size_t)w.K * w.H + 1;
  b.stats = (int64_t*)((char*)w.h_back + ((off32 * sizeof(int32_t) + 7) & ~(size_t)7));
  return b;
}

static agnes_status wait_prepared(agnes_ctx* ctx) {
  if (!ctx) return AGNES_EINVAL;
  if (!ctx->prepared) {
    set_err(ctx, "no hyperbatch has been prepared");
    return AGNES_ESTATE;
  }
  if (!ctx->synced) {
    cudaSetDevice(ctx->device);
    cudaError_t e = cudaEventSynchronize(ctx->done);
    if (e != cudaSuccess) {
      set_err(ctx, "waiting for the hyperbatch failed: %s", cudaGetErrorString(e));
      return AGNES_ECUDA;
    }
    ctx->synced = true;
  }
  const Back b = back_of(ctx->ws);
  const int32_t s = *b.status;
  if (s != 0) {
    if (s & kErrTargetRange) {
      set_err(ctx, "a target id is outside [0, %lld)", (long long)ctx->N);
      return AGNES_EINVAL;
    }
    if (s & kErrTargetDup) {
      set_err(ctx, "a target id is repeated within a minibatch");
      return AGNES_EINVAL;
    }
    set_err(ctx, "device status word 0x%x", s);
    return AGNES_EKERNEL;
  }
  return AGNES_OK;
}

// ============================================================================
// Public API
// ============================================================================

static void drop_launch_graph(agnes_ctx::LaunchGraph* g) {
  if (g->exec) cudaGraphExecDestroy(g->exec);
  if (g->graph) cudaGraphDestroy(g->graph);
  g->exec = nullptr;
  g->graph = nullptr;
  g->n_marks = 0;
}

extern "C" {

const char* agnes_status_string(agnes_status s) {
  switch (s) {
    case AGNES_OK: return "ok";
    case AGNES_EINVAL: return "invalid argument";
    case AGNES_ERANGE: return "size out of range";
    case AGNES_ENOMEM: return "out of memory";
    case AGNES_ECUDA: return "CUDA error";
    case AGNES_ESTATE: return "call out of order";
    case AGNES_ETIMEOUT: return "timed out";
    case AGNES_EKERNEL: return "kernel reported an inconsistency";
  }
  return "unknown status";
}

const char* agnes_last_error(agnes_ctx* ctx) { return ctx ? ctx->err : g_err; }

agnes_status agnes_free(agnes_ctx* ctx) {
  if (!ctx) return AGNES_OK;
  cudaSetDevice(ctx->device);
  cudaDeviceSynchronize();
  drop_launch_graph(&ctx->lg);
  if (ctx->lg.cap) cudaStreamDestroy(ctx->lg.cap);
  free_workspace(&ctx->ws);
  free_block_tables(&ctx->bt);
  if (ctx->own_offsets) cudaFree(ctx->offsets);
  if (ctx->own_indices) cudaFree(ctx->indices);
  if (ctx->own_features) cudaFree(ctx->features);
  if (ctx->done) cudaEventDestroy(ctx->done);
  for (int i = 0; i < kStreamSlots; ++i) {
    if (ctx->slot_copied[i]) cudaEventDestroy(ctx->slot_copied[i]);
    if (ctx->slot_free[i]) cudaEventDestroy(ctx->slot_free[i]);
  }
  if (ctx->copy_stream) cudaStreamDestroy(ctx->copy_stream);
  cudaFree(ctx->slots);
  cudaFree(ctx->d_touched);
  cudaFree(ctx->d_counts);
  cudaFree(ctx->d_src);
  cudaFree(ctx->scratch);
  if (ctx->pinned) cudaFreeHost(ctx->pinned);
  cudaFree(ctx->d_job_blk);
  cudaFree(ctx->d_job_dst);
  cudaFree(ctx->d_addr);
  cudaFree(ctx->rm_bitmap);
  cudaFree(ctx->rm_wpref);
  cudaFree(ctx->rm_dcnt);
  cudaFree(ctx->rm_doff);
  cudaFree(ctx->rm_staging);
  cudaFree(ctx->d_host_rows);
  if (ctx->h_rm) cudaFreeHost(ctx->h_rm);
  cudaFree(ctx->fcache);
  if (ctx->gather_start) cudaEventDestroy(ctx->gather_start);
  if (ctx->h_counts) cudaFreeHost(ctx->h_counts);
  if (ctx->h_touched) cudaFreeHost(ctx->h_touched);
  if (ctx->h_src) cudaFreeHost(ctx->h_src);
  if (ctx->h_job_blk) cudaFreeHost(ctx->h_job_blk);
  if (ctx->h_job_dst) cudaFreeHost(ctx->h_job_dst);
  if (ctx->h_addr) cudaFreeHost(ctx->h_addr);
  {
    agnes_ctx::Topo& tp = ctx->topo;
    if (tp.copy) cudaStreamDestroy(tp.copy);
    if (tp.uploaded) cudaEventDestroy(tp.uploaded);
    for (int i = 0; i < 2; ++i)
      if (tp.wave_done[i]) cudaEventDestroy(tp.wave_done[i]);
    cudaFree(tp.d_jobs);
    if (tp.h_jobs) cudaFreeHost(tp.h_jobs);
    cudaFree(tp.gbuf);
    cudaFree(tp.d_slot);
    cudaFree(tp.d_need);
    if (tp.h_slot_stage) cudaFreeHost(tp.h_slot_stage);
    if (tp.h_need) cudaFreeHost(tp.h_need);
    cudaFree(tp.d_acc);
    cudaFree(tp.d_cached);
    if (tp.h_acc) cudaFreeHost(tp.h_acc);
    if (tp.h_cached) cudaFreeHost(tp.h_cached);
  }
  if (ctx->ev_created)
    for (int r = 0; r < kEventRing; ++r)
      for (int i = 0; i <= kMaxPhases; ++i) cudaEventDestroy(ctx->ev[r][i]);
  delete ctx;
  return AGNES_OK;
}

static agnes_status adopt_or_copy(agnes_ctx* ctx, const void* src, size_t bytes, void** dst,
                                  bool* own, cudaStream_t st) {
  if (is_device_ptr(src)) {
    *dst = const_cast<void*>(src);
    *own = false;
    return AGNES_OK;
  }
  CK(ctx, cudaMalloc(dst, bytes ? bytes : 1));
  *own = true;
  CK(ctx, cudaMemcpyAsync(*dst, src, bytes, cudaMemcpyHostToDevice, st));
  return AGNES_OK;
}

// Staging ring (block mode), feature cache, copy stream and host tables for
// host-resident features.
static agnes_status setup_streaming(agnes_ctx* ctx, const agnes_graph_desc* d, cudaStream_t st) {
  const int64_t nfb = ctx->bt.n_feat_blocks;
  const int64_t blk = ctx->bt.rows_per_feat_block * ctx->row_bytes;
  {
    void* dv = nullptr;
    CK(ctx, cudaHostGetDevicePointer(&dv, ctx->features, 0));
    ctx->features_dev = (const char*)dv;
  }
  CK(ctx, cudaStreamCreateWithFlags(&ctx->copy_stream, cudaStreamNonBlocking));
  for (int i = 0; i < kStreamSlots; ++i) {
    CK(ctx, cudaEventCreateWithFlags(&ctx->slot_copied[i], cudaEventDisableTiming));
    CK(ctx, cudaEventCreateWithFlags(&ctx->slot_free[i], cudaEventDisableTiming));
  }
  CK(ctx, cudaEventCreateWithFlags(&ctx->gather_start, cudaEventDisableTiming));
  if (ctx->feature_io == AGNES_FEATURE_IO_BLOCKS) {
    ctx->slot_bytes = (int64_t)kStreamBatchBlocks * blk;
    CK(ctx, cudaMalloc((void**)&ctx->slots, (size_t)(ctx->slot_bytes * kStreamSlots)));
  } else {
    const size_t T = (size_t)ctx->bt.T;
    CK(ctx, cudaMalloc((void**)&ctx->rm_bitmap, sizeof(uint32_t) * T * kTileWords));
    CK(ctx, cudaMalloc((void**)&ctx->rm_wpref, sizeof(uint16_t) * T * kTileWords));
    CK(ctx, cudaMalloc((void**)&ctx->rm_dcnt, sizeof(int32_t) * T));
    CK(ctx, cudaMalloc((void**)&ctx->rm_doff, sizeof(int32_t) * (T + 1)));
    CK(ctx, cudaMalloc((void**)&ctx->d_host_rows, sizeof(unsigned long long)));
    CK(ctx, cudaMallocHost((void**)&ctx->h_rm, sizeof(int64_t) * 2));
    ctx->h_rm[0] = ctx->h_rm[1] = 0;
  }
  const size_t n1 = (size_t)(nfb + 1);
  CK(ctx, cudaMalloc((void**)&ctx->d_touched, sizeof(int32_t) * n1));
  CK(ctx, cudaMalloc((void**)&ctx->d_counts, sizeof(int32_t) * n1));
  CK(ctx, cudaMalloc((void**)&ctx->d_src, sizeof(unsigned long long) * n1));
  CK(ctx, cudaMalloc((void**)&ctx->d_job_blk, sizeof(int32_t) * n1));
  CK(ctx, cudaMalloc((void**)&ctx->d_job_dst, sizeof(unsigned long long) * n1));
  CK(ctx, cudaMalloc((void**)&ctx->d_addr, sizeof(unsigned long long) * n1));
  CK(ctx, cudaMallocHost((void**)&ctx->h_counts, sizeof(int32_t) * n1));
  CK(ctx, cudaMallocHost((void**)&ctx->h_touched, sizeof(int32_t) * n1));
  CK(ctx, cudaMallocHost((void**)&ctx->h_src, sizeof(unsigned long long) * n1));
  CK(ctx, cudaMallocHost((void**)&ctx->h_job_blk, sizeof(int32_t) * n1));
  CK(ctx, cudaMallocHost((void**)&ctx->h_job_dst, sizeof(unsigned long long) * n1));
  CK(ctx, cudaMallocHost((void**)&ctx->h_addr, sizeof(unsigned long long) * n1));
  ctx->fblock_first_tile.resize(n1);
  CK(ctx, cudaMemcpyAsync(ctx->fblock_first_tile.data(), ctx->bt.fblock_first_tile,
                          sizeof(int32_t) * n1, cudaMemcpyDeviceToHost, st));
  ctx->fcache_slots = d->feature_cache_bytes > 0 ? d->feature_cache_bytes / blk : 0;
  if (ctx->fcache_slots > nfb) ctx->fcache_slots = nfb;
  ctx->fcache_threshold = d->feature_cache_threshold;
  if (ctx->fcache_slots > 0)
    CK(ctx, cudaMalloc((void**)&ctx->fcache, (size_t)(ctx->fcache_slots * blk)));
  ctx->acc.assign((size_t)nfb, 0);
  ctx->cslot_of.assign((size_t)nfb, -1);
  ctx->cblock_of.assign((size_t)ctx->fcache_slots, -1);
  ctx->cresident.assign((size_t)ctx->fcache_slots, 0);
  CK(ctx, cudaStreamSynchronize(st));
  return AGNES_OK;
}

// Graph buffer, tables and copy stream for topology in pinned host memory.
// Host copies of the block tables the topology modes plan with: the edge
// range of every physical block and the blocks of every block run.
static agnes_status topology_host_tables(agnes_ctx* ctx, const agnes_graph_desc* d,
                                         cudaStream_t st) {
  agnes_ctx::Topo& tp = ctx->topo;
  const int64_t nb = ctx->bt.n_blocks, ns = ctx->bt.n_starts;
  tp.host_indices = d->indices;
  tp.epb = d->adj_block_bytes / 4;
  tp.e0.resize((size_t)nb);
  tp.e1.resize((size_t)nb);
  tp.start_block.resize((size_t)ns + 1);
  tp.run_first_tile.resize((size_t)ns + 1);
  CK(ctx, cudaMemcpyAsync(tp.e0.data(), ctx->bt.blk_e0, sizeof(int64_t) * nb,
                          cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaMemcpyAsync(tp.e1.data(), ctx->bt.blk_e1, sizeof(int64_t) * nb,
                          cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaMemcpyAsync(tp.start_block.data(), ctx->bt.start_block, sizeof(int32_t) * ns,
                          cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaMemcpyAsync(tp.run_first_tile.data(), ctx->bt.run_first_tile,
                          sizeof(int32_t) * (ns + 1), cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaStreamSynchronize(st));
  tp.start_block[(size_t)ns] = (int32_t)nb;
  return AGNES_OK;
}

// A topology cache for in-place reads: graph_buffer_bytes / adj_block_bytes
// slots, filled between hyperbatches with the block runs the frontiers
// requested most (update_topology_cache).
static agnes_status setup_topology_cache(agnes_ctx* ctx, const agnes_graph_desc* d,
                                         cudaStream_t st) {
  agnes_ctx::Topo& tp = ctx->topo;
  agnes_status rc = topology_host_tables(ctx, d, st);
  if (rc != AGNES_OK) return rc;
  const int64_t nb = ctx->bt.n_blocks, ns = ctx->bt.n_starts;
  tp.slots = d->graph_buffer_bytes / d->adj_block_bytes;
  if (tp.slots > nb) tp.slots = nb;
  if (tp.slots < 1) return AGNES_OK;
  tp.cache = true;
  tp.dev_view = ctx->indices;  // the device view of the host neighbour lists
  CK(ctx, cudaMalloc((void**)&tp.gbuf, sizeof(int32_t) * (size_t)(tp.slots * tp.epb)));
  CK(ctx, cudaMalloc((void**)&tp.d_slot, sizeof(int32_t) * (size_t)nb));
  CK(ctx, cudaMallocHost((void**)&tp.h_slot_stage, sizeof(int32_t) * (size_t)nb));
  CK(ctx, cudaMemsetAsync(tp.d_slot, 0xff, sizeof(int32_t) * (size_t)nb, st));
  CK(ctx, cudaMalloc((void**)&tp.d_acc, sizeof(unsigned long long) * (size_t)ns));
  CK(ctx, cudaMallocHost((void**)&tp.h_acc, sizeof(unsigned long long) * (size_t)ns));
  CK(ctx, cudaMalloc((void**)&tp.d_cached, sizeof(unsigned long long)));
  CK(ctx, cudaMallocHost((void**)&tp.h_cached, sizeof(unsigned long long)));
  CK(ctx, cudaMemsetAsync(tp.d_acc, 0, sizeof(unsigned long long) * (size_t)ns, st));
  CK(ctx, cudaMemsetAsync(tp.d_cached, 0, sizeof(unsigned long long), st));
  *tp.h_cached = 0;
  tp.jobs_cap = (int32_t)tp.slots;
  CK(ctx, cudaMalloc((void**)&tp.d_jobs, sizeof(int2) * (size_t)tp.jobs_cap));
  CK(ctx, cudaMallocHost((void**)&tp.h_jobs, sizeof(int2) * (size_t)tp.jobs_cap));
  tp.slot_of.assign((size_t)nb, -1);
  tp.block_of.assign((size_t)tp.slots, -1);
  tp.run_of.resize((size_t)nb);
  for (int64_t r = 0; r < ns; ++r)
    for (int32_t b = tp.start_block[(size_t)r]; b < tp.start_block[(size_t)r + 1]; ++b)
      tp.run_of[(size_t)b] = (int32_t)r;
  CK(ctx, cudaStreamSynchronize(st));
  return AGNES_OK;
}

static agnes_status setup_topology(agnes_ctx* ctx, const agnes_graph_desc* d, cudaStream_t st) {
  agnes_ctx::Topo& tp = ctx->topo;
  const int64_t nb = ctx->bt.n_blocks, ns = ctx->bt.n_starts;
  agnes_status rc = topology_host_tables(ctx, d, st);
  if (rc != AGNES_OK) return rc;
  tp.on = true;
  int64_t longest = 1;
  for (int64_t r = 0; r < ns; ++r) {
    const int64_t m = tp.start_block[(size_t)r + 1] - tp.start_block[(size_t)r];
    if (m > longest) longest = m;
  }
  tp.slots = d->graph_buffer_bytes > 0 ? d->graph_buffer_bytes / d->adj_block_bytes : nb;
  if (tp.slots > nb) tp.slots = nb;
  if (tp.slots < 2 * longest) {
    set_err(ctx, "graph_buffer_bytes holds %lld blocks; two waves of the largest object need %lld",
            (long long)tp.slots, (long long)(2 * longest));
    return AGNES_EINVAL;
  }
  CK(ctx, cudaMalloc((void**)&tp.gbuf, sizeof(int32_t) * (size_t)(tp.slots * tp.epb)));
  CK(ctx, cudaMalloc((void**)&tp.d_slot, sizeof(int32_t) * (size_t)nb));
  CK(ctx, cudaMalloc((void**)&tp.d_need, (size_t)ns + 1));
  CK(ctx, cudaMallocHost((void**)&tp.h_slot_stage, sizeof(int32_t) * (size_t)nb));
  CK(ctx, cudaMallocHost((void**)&tp.h_need, (size_t)ns + 1));
  CK(ctx, cudaMemsetAsync(tp.d_slot, 0xff, sizeof(int32_t) * (size_t)nb, st));
  CK(ctx, cudaStreamCreateWithFlags(&tp.copy, cudaStreamNonBlocking));
  CK(ctx, cudaEventCreateWithFlags(&tp.uploaded, cudaEventDisableTiming));
  for (int i = 0; i < 2; ++i)
    CK(ctx, cudaEventCreateWithFlags(&tp.wave_done[i], cudaEventDisableTiming));
  {
    void* dv = nullptr;
    CK(ctx, cudaHostGetDevicePointer(&dv, const_cast<int32_t*>(d->indices), 0));
    tp.dev_view = (const int32_t*)dv;
  }
  tp.jobs_cap = (int32_t)(tp.slots < nb ? tp.slots : nb);
  CK(ctx, cudaMalloc((void**)&tp.d_jobs, sizeof(int2) * (size_t)tp.jobs_cap));
  CK(ctx, cudaMallocHost((void**)&tp.h_jobs, sizeof(int2) * (size_t)tp.jobs_cap));
  tp.slot_of.assign((size_t)nb, -1);
  tp.block_of.assign((size_t)tp.slots, -1);
  tp.pinned.assign((size_t)tp.slots, 0);
  tp.prev.resize((size_t)tp.slots);
  tp.next.resize((size_t)tp.slots);
  for (int64_t i = 0; i < tp.slots; ++i) {  // all slots free, in LRU order
    tp.prev[(size_t)i] = (int32_t)i - 1;
    tp.next[(size_t)i] = i + 1 < tp.slots ? (int32_t)i + 1 : -1;
  }
  tp.head = 0;
  tp.tail = (int32_t)tp.slots - 1;
  CK(ctx, cudaStreamSynchronize(st));
  return AGNES_OK;
}

// LRU list: move slot i to the most-recent end.
static void lru_touch(agnes_ctx::Topo& tp, int32_t i) {
  if (tp.tail == i) return;
  const int32_t p = tp.prev[(size_t)i], n = tp.next[(size_t)i];
  if (p >= 0) tp.next[(size_t)p] = n; else tp.head = n;
  if (n >= 0) tp.prev[(size_t)n] = p;
  tp.prev[(size_t)i] = tp.tail;
  tp.next[(size_t)i] = -1;
  tp.next[(size_t)tp.tail] = i;
  tp.tail = i;
}

agnes_status agnes_load_graph(const agnes_graph_desc* d, int device, void* cuda_stream,
                              agnes_ctx** out) {
  if (!out) {
    set_err(nullptr, "out is NULL");
    return AGNES_EINVAL;
  }
  *out = nullptr;
  if (!d) {
    set_err(nullptr, "desc is NULL");
    return AGNES_EINVAL;
  }
  if (d->num_nodes < 1 || d->num_nodes >= ((int64_t)1 << 31)) {
    set_err(nullptr, "num_nodes must be in [1, 2^31)");
    return d->num_nodes < 1 ? AGNES_EINVAL : AGNES_ERANGE;
  }
  if (d->offsets_bits != 32 && d->offsets_bits != 64) {
    set_err(nullptr, "offsets_bits must be 32 or 64");
    return AGNES_EINVAL;
  }
  if (d->num_edges < 0 || (d->offsets_bits == 32 && d->num_edges >= ((int64_t)1 << 31))) {
    set_err(nullptr, "num_edges out of range for the offsets type");
    return AGNES_ERANGE;
  }
  if (d->topology_on_host && (!d->indices || !is_pinned_host_ptr(d->indices))) {
    set_err(nullptr, "topology_on_host requires indices in pinned host memory");
    return AGNES_EINVAL;
  }
  if (!d->offsets || (d->num_edges > 0 && !d->indices) || !d->features) {
    set_err(nullptr, "offsets, indices and features must be non-NULL");
    return AGNES_EINVAL;
  }
  if (d->feat_dtype != AGNES_F32 && d->feat_dtype != AGNES_F16) {
    set_err(nullptr, "feat_dtype must be AGNES_F32 or AGNES_F16");
    return AGNES_EINVAL;
  }
  const int64_t esize = d->feat_dtype == AGNES_F32 ? 4 : 2;
  if (d->feat_dim < 1 || d->feat_dim > (1 << 20)) {
    set_err(nullptr, "feat_dim must be in [1, 2^20]");
    return AGNES_EINVAL;
  }
  const int64_t row_bytes = d->feat_dim * esize;
  if (d->adj_block_bytes < 64 || d->adj_block_bytes > ((int64_t)1 << 34)) {
    set_err(nullptr, "adj_block_bytes must be in [64, 2^34]");
    return AGNES_EINVAL;
  }
  if (d->feat_block_bytes < row_bytes || d->feat_block_bytes > ((int64_t)1 << 34)) {
    set_err(nullptr, "feat_block_bytes must hold at least one feature row");
    return AGNES_EINVAL;
  }
  if (d->features_on_host && !is_pinned_host_ptr(d->features)) {
    set_err(nullptr, "features_on_host requires pinned host memory");
    return AGNES_EINVAL;
  }
  if (d->features_on_host && (row_bytes % 16) != 0) {
    set_err(nullptr, "features_on_host needs feature rows of a multiple of 16 bytes");
    return AGNES_EINVAL;
  }
  if (d->features_on_host && ((uintptr_t)d->features % 16) != 0) {
    set_err(nullptr, "features_on_host needs a 16-byte aligned feature matrix");
    return AGNES_EINVAL;
  }
  if (d->topology_io != AGNES_TOPOLOGY_IO_BLOCKS && d->topology_io != AGNES_TOPOLOGY_IO_ROWS) {
    set_err(nullptr, "topology_io must be AGNES_TOPOLOGY_IO_BLOCKS or AGNES_TOPOLOGY_IO_ROWS");
    return AGNES_EINVAL;
  }
  if (d->feature_io != AGNES_FEATURE_IO_BLOCKS && d->feature_io != AGNES_FEATURE_IO_ROWS) {
    set_err(nullptr, "feature_io must be AGNES_FEATURE_IO_BLOCKS or AGNES_FEATURE_IO_ROWS");
    return AGNES_EINVAL;
  }
  if (d->feature_cache_bytes < 0 || d->feature_cache_threshold < 0 ||
      (d->feature_cache_bytes > 0 && !d->features_on_host)) {
    set_err(nullptr, "feature_cache_bytes and feature_cache_threshold must be >= 0, and a "
                     "feature cache needs features_on_host");
    return AGNES_EINVAL;
  }
  if (cudaSetDevice(device) != cudaSuccess) {
    cudaGetLastError();
    set_err(nullptr, "invalid device %d", device);
    return AGNES_EINVAL;
  }
  agnes_ctx* ctx = new (std::nothrow) agnes_ctx();
  if (!ctx) {
    set_err(nullptr, "out of host memory");
    return AGNES_ENOMEM;
  }
  ctx->device = device;
  cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, device);
  if (ctx->num_sms < 1) ctx->num_sms = 1;
  ctx->N = d->num_nodes;
  ctx->E = d->num_edges;
  ctx->offsets_bits = d->offsets_bits;
  ctx->feat_dtype = d->feat_dtype;
  ctx->feat_dim = d->feat_dim;
  ctx->row_bytes = row_bytes;
  ctx->features_on_host = d->features_on_host;
  ctx->feature_io = d->feature_io;
  ctx->adj_block_bytes = d->adj_block_bytes;
  ctx->feat_block_bytes = d->feat_block_bytes;
  cudaStream_t st = (cudaStream_t)cuda_stream;

  agnes_status rc;
  const size_t off_bytes = (size_t)(d->num_nodes + 1) * (d->offsets_bits / 8);
  rc = adopt_or_copy(ctx, d->offsets, off_bytes, &ctx->offsets, &ctx->own_offsets, st);
  if (rc == AGNES_OK && d->num_edges > 0 && !d->topology_on_host)
    rc = adopt_or_copy(ctx, d->indices, (size_t)d->num_edges * 4, (void**)&ctx->indices,
                       &ctx->own_indices, st);
  if (rc == AGNES_OK && d->num_edges > 0 && d->topology_on_host &&
      d->topology_io == AGNES_TOPOLOGY_IO_ROWS) {
    // the sampler reads neighbour entries in place, through the device view
    void* dv = nullptr;
    if (cudaHostGetDevicePointer(&dv, const_cast<int32_t*>(d->indices), 0) != cudaSuccess) {
      cudaGetLastError();
      set_err(ctx, "cudaHostGetDevicePointer failed for the host neighbour lists");
      rc = AGNES_ECUDA;
    } else {
      ctx->indices = (int32_t*)dv;
      ctx->own_indices = false;
    }
  }
  if (rc == AGNES_OK) {
    if (d->features_on_host) {
      ctx->features = const_cast<void*>(d->features);
      ctx->own_features = false;
    } else {
      rc = adopt_or_copy(ctx, d->features, (size_t)(d->num_nodes * row_bytes), &ctx->features,
                         &ctx->own_features, st);
    }
  }
  if (rc == AGNES_OK) {
    int64_t ends[2] = {0, 0};
    cudaError_t e;
    if (d->offsets_bits == 32) {
      int32_t v[2];
      e = cudaMemcpyAsync(&v[0], ctx->offsets, 4, cudaMemcpyDeviceToHost, st);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(&v[1], (int32_t*)ctx->offsets + d->num_nodes, 4,
                            cudaMemcpyDeviceToHost, st);
      if (e == cudaSuccess) e = cudaStreamSynchronize(st);
      ends[0] = v[0];
      ends[1] = v[1];
    } else {
      e = cudaMemcpyAsync(&ends[0], ctx->offsets, 8, cudaMemcpyDeviceToHost, st);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(&ends[1], (int64_t*)ctx->offsets + d->num_nodes, 8,
                            cudaMemcpyDeviceToHost, st);
      if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    }
    if (e != cudaSuccess) {
      set_err(ctx, "reading offsets failed: %s", cudaGetErrorString(e));
      rc = AGNES_ECUDA;
    } else if (ends[0] != 0 || ends[1] != d->num_edges) {
      set_err(ctx, "offsets[0] must be 0 and offsets[N] must equal num_edges");
      rc = AGNES_EINVAL;
    }
  }
  if (rc == AGNES_OK) {
    const int64_t rpb = d->feat_block_bytes / row_bytes;
    cudaError_t e = build_block_tables(ctx->offsets, d->offsets_bits, d->num_nodes, d->num_edges,
                                       d->adj_block_bytes, rpb, &ctx->bt, st, ctx->err,
                                       sizeof(ctx->err));
    if (e != cudaSuccess) rc = e == cudaErrorMemoryAllocation ? AGNES_ENOMEM : AGNES_ECUDA;
  }
  if (rc == AGNES_OK && d->features_on_host) rc = setup_streaming(ctx, d, st);
  if (rc == AGNES_OK && d->topology_on_host && d->num_edges > 0 &&
      d->topology_io == AGNES_TOPOLOGY_IO_BLOCKS)
    rc = setup_topology(ctx, d, st);
  if (rc == AGNES_OK && d->topology_on_host && d->num_edges > 0 &&
      d->topology_io == AGNES_TOPOLOGY_IO_ROWS && d->graph_buffer_bytes > 0)
    rc = setup_topology_cache(ctx, d, st);
  if (rc == AGNES_OK && cudaEventCreateWithFlags(&ctx->done, cudaEventDisableTiming) != cudaSuccess) {
    set_err(ctx, "cudaEventCreate failed");
    rc = AGNES_ECUDA;
  }
  if (rc != AGNES_OK) {
    snprintf(g_err, sizeof(g_err), "%s", ctx->err);
    agnes_free(ctx);
    return rc;
  }
  *out = ctx;
  return AGNES_OK;
}

// Sampling with the topology in pinned host memory.  The block runs the
// frontier touches are read back; runs are taken in ascending order into
// waves that fit the graph buffer: each needed block is either resident
// (a hit: pinned and moved to the recent end of the LRU list) or copied into
// the least recently used unpinned slot on the side stream.  The slot table
// is uploaded, the wave's cells are sampled, and the wave's blocks unpin when
// the next wave starts (its copies wait for this wave's sampling to finish).
static agnes_status fill_streamed(agnes_ctx* ctx, const HopArgs& a, int cur, int h,
                                  cudaStream_t st) {
  Workspace& w = ctx->ws;
  agnes_ctx::Topo& tp = ctx->topo;
  const int64_t ns = ctx->bt.n_starts, nb = ctx->bt.n_blocks;
  const int32_t H = w.H, T = (int32_t)ctx->bt.T;
  // a wave may use half the buffer: the previous wave's blocks stay pinned
  // while it samples, so the next wave's blocks load at the same time
  const int64_t wave_cap = tp.slots / 2;
  CK(ctx, launch_mark_runs(w.fcell_off[cur], T, H, ctx->bt.tile_adj_start, tp.d_need, ns, w.status,
                           st));
  CK(ctx, cudaMemcpyAsync(tp.h_need, tp.d_need, (size_t)ns, cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaStreamSynchronize(st));
  // Hops sweep their block runs in alternating directions, so each hop
  // starts on the blocks the previous one used last -- the ones LRU kept.
  // (The order of a hop's blocks does not change any result.)
  const int64_t step = (tp.sweeps++ & 1) ? -1 : 1;
  auto inside = [&](int64_t x) { return x >= 0 && x < ns; };
  int64_t r = step > 0 ? 0 : ns - 1;
  while (inside(r) && !tp.h_need[r]) r += step;
  while (inside(r)) {
    // the staging buffers (jobs, slot table) are rewritten below: wait until
    // the previous wave's upload and loads have consumed them
    if (tp.uploaded_used) CK(ctx, cudaEventSynchronize(tp.uploaded));
    tp.wave += 1;
    const uint32_t wave = tp.wave;
    int64_t pinned_now = 0;
    int32_t njobs = 0;
    int64_t r_lo = r, r_hi = r;  // the wave's runs, [r_lo, r_hi]
    while (inside(r)) {
      if (!tp.h_need[r]) {
        r += step;
        continue;
      }
      const int32_t b0 = tp.start_block[(size_t)r], b1 = tp.start_block[(size_t)r + 1];
      if (pinned_now > 0 && pinned_now + (b1 - b0) > wave_cap) break;  // wave full
      for (int32_t b = b0; b < b1; ++b) {
        int32_t sl = tp.slot_of[(size_t)b];
        if (sl >= 0) {
          tp.hits += 1;
        } else {
          // least recently used slot not pinned by this wave or the previous one
          sl = tp.head;
          while (sl >= 0 && tp.pinned[(size_t)sl] + 1 >= wave) sl = tp.next[(size_t)sl];
          if (sl < 0) {
            set_err(ctx, "graph buffer exhausted inside a wave");
            return AGNES_EKERNEL;
          }
          const int32_t old = tp.block_of[(size_t)sl];
          if (old >= 0) tp.slot_of[(size_t)old] = -1;
          tp.block_of[(size_t)sl] = b;
          tp.slot_of[(size_t)b] = sl;
          tp.h_jobs[njobs++] = make_int2(b, sl);
          tp.loaded_blocks += 1;
          tp.loaded_bytes += sizeof(int32_t) * (tp.e1[(size_t)b] - tp.e0[(size_t)b]);
        }
        tp.pinned[(size_t)sl] = wave;
        lru_touch(tp, sl);
        ++pinned_now;
      }
      r_lo = r < r_lo ? r : r_lo;
      r_hi = r > r_hi ? r : r_hi;
      r += step;
    }
    // the slots taken now were last read by wave - 2 at the latest
    CK(ctx, cudaStreamWaitEvent(tp.copy, tp.wave_done[wave & 1], 0));
    memcpy(tp.h_slot_stage, tp.slot_of.data(), sizeof(int32_t) * (size_t)nb);
    CK(ctx, cudaMemcpyAsync(tp.d_slot, tp.h_slot_stage, sizeof(int32_t) * (size_t)nb,
                            cudaMemcpyHostToDevice, tp.copy));
    if (njobs > 0) {
      CK(ctx, cudaMemcpyAsync(tp.d_jobs, tp.h_jobs, sizeof(int2) * (size_t)njobs,
                              cudaMemcpyHostToDevice, tp.copy));
      CK(ctx, launch_load_blocks(tp.dev_view, ctx->bt.blk_e0, ctx->bt.blk_e1, tp.d_jobs, njobs,
                                 tp.gbuf, tp.epb, ctx->num_sms, tp.copy));
    }
    CK(ctx, cudaEventRecord(tp.uploaded, tp.copy));
    tp.uploaded_used = true;
    CK(ctx, cudaStreamWaitEvent(st, tp.uploaded, 0));
    FillRange fr;
    fr.cell_lo = (int64_t)tp.run_first_tile[(size_t)r_lo] * H;
    fr.cell_hi = (int64_t)tp.run_first_tile[(size_t)r_hi + 1] * H;
    fr.tile_adj_block = ctx->bt.tile_adj_block;
    fr.blk_slot = tp.d_slot;
    fr.blk_e0 = ctx->bt.blk_e0;
    fr.gbuf = tp.gbuf;
    fr.epb = tp.epb;
    fr.bb = ctx->adj_block_bytes;
    CK(ctx, launch_sample_fill(a, w.fb_id[cur], w.fb_pos[cur], w.fcell_off[cur], w.indptr[h], w.nbr,
                               w.scnt, w.scell, w.srank, fr, ctx->num_sms, st));
    CK(ctx, cudaEventRecord(tp.wave_done[wave & 1], st));
    tp.waves += 1;
    while (inside(r) && !tp.h_need[r]) r += step;
  }
  return AGNES_OK;
}

// Bytes of feature block b (the last block of the matrix may be short).
static int64_t feat_block_bytes_of(const agnes_ctx* ctx, int32_t b) {
  const int64_t rpb = ctx->bt.rows_per_feat_block;
  const int64_t r0 = (int64_t)b * rpb;
  const int64_t r1 = r0 + rpb < ctx->N ? r0 + rpb : ctx->N;
  return (r1 - r0) * ctx->row_bytes;
}

// Block mode (Sec. 3.3 block-wise I/O, Sec. 3.4 (4) asynchronous I/O, the
// host link standing in for the SSD).  A touched block that is cached and
// resident is read in place; one admitted to the cache but not yet loaded is
// loaded into its cache slot; any other is loaded into the ring of HBM
// staging slots.  Batch by batch, a loader kernel on the side stream reads
// the batch's blocks over the host link; the batch's gather waits for it and
// the next load into a slot waits for the gather that last read it.
static agnes_status gather_blocks_io(agnes_ctx* ctx, int cur, int32_t n, int64_t* bytes_out,
                                     int64_t* hits_out, cudaStream_t st) {
  Workspace& w = ctx->ws;
  const int64_t rpb = ctx->bt.rows_per_feat_block;
  const int64_t rb = ctx->row_bytes;
  const int64_t blk = rpb * rb;
  const int32_t H = w.H;
  const int32_t nbatch = (n + kStreamBatchBlocks - 1) / kStreamBatchBlocks;
  std::vector<int32_t> job0((size_t)nbatch + 1, 0);
  int32_t nj = 0;
  int64_t bytes = 0, hits = 0;
  for (int32_t batch = 0; batch < nbatch; ++batch) {
    const int32_t i0 = batch * kStreamBatchBlocks;
    const int32_t i1 = i0 + kStreamBatchBlocks < n ? i0 + kStreamBatchBlocks : n;
    char* slot = ctx->slots + (int64_t)(batch % kStreamSlots) * ctx->slot_bytes;
    job0[(size_t)batch] = nj;
    int32_t p = 0;
    for (int32_t i = i0; i < i1; ++i) {
      const int32_t b = ctx->h_touched[i];
      const int32_t cs = ctx->fcache_slots ? ctx->cslot_of[(size_t)b] : -1;
      unsigned long long a;
      bool load = true;
      if (cs >= 0) {
        a = (unsigned long long)(uintptr_t)(ctx->fcache + (int64_t)cs * blk);
        if (ctx->cresident[(size_t)cs]) {
          load = false;
          hits += 1;
        } else {
          ctx->cresident[(size_t)cs] = 1;
          ctx->fcache_loads += 1;
        }
      } else {
        a = (unsigned long long)(uintptr_t)(slot + (int64_t)p++ * blk);
      }
      ctx->h_src[i] = a;
      if (load) {
        ctx->h_job_blk[nj] = b;
        ctx->h_job_dst[nj] = a;
        ++nj;
        bytes += feat_block_bytes_of(ctx, b);
      }
    }
  }
  job0[(size_t)nbatch] = nj;
  if (n > 0) {
    CK(ctx, cudaMemcpyAsync(ctx->d_touched, ctx->h_touched, sizeof(int32_t) * n,
                            cudaMemcpyHostToDevice, st));
    CK(ctx, cudaMemcpyAsync(ctx->d_src, ctx->h_src, sizeof(unsigned long long) * n,
                            cudaMemcpyHostToDevice, st));
  }
  if (nj > 0) {
    CK(ctx, cudaMemcpyAsync(ctx->d_job_blk, ctx->h_job_blk, sizeof(int32_t) * nj,
                            cudaMemcpyHostToDevice, st));
    CK(ctx, cudaMemcpyAsync(ctx->d_job_dst, ctx->h_job_dst, sizeof(unsigned long long) * nj,
                            cudaMemcpyHostToDevice, st));
  }
  // the job tables are on the device, and cache slots are no longer read by
  // earlier gathers, once st reaches this point
  CK(ctx, cudaEventRecord(ctx->gather_start, st));
  CK(ctx, cudaStreamWaitEvent(ctx->copy_stream, ctx->gather_start, 0));
  for (int32_t batch = 0; batch < nbatch; ++batch) {
    const int32_t i0 = batch * kStreamBatchBlocks;
    const int32_t nb = n - i0 < kStreamBatchBlocks ? n - i0 : kStreamBatchBlocks;
    const int s = batch % kStreamSlots;
    if (ctx->slot_used[s]) CK(ctx, cudaStreamWaitEvent(ctx->copy_stream, ctx->slot_free[s], 0));
    const int32_t j0 = job0[(size_t)batch], j1 = job0[(size_t)batch + 1];
    CK(ctx, launch_load_feat_blocks(ctx->features_dev, ctx->N * rb, ctx->d_job_blk + j0,
                                    ctx->d_job_dst + j0, j1 - j0, blk, ctx->num_sms,
                                    ctx->copy_stream));
    CK(ctx, cudaEventRecord(ctx->slot_copied[s], ctx->copy_stream));
    CK(ctx, cudaStreamWaitEvent(st, ctx->slot_copied[s], 0));
    const int64_t cell_lo = (int64_t)ctx->fblock_first_tile[ctx->h_touched[i0]] * H;
    const int64_t cell_hi = (int64_t)ctx->fblock_first_tile[ctx->h_touched[i0 + nb - 1] + 1] * H;
    CK(ctx, launch_gather_staged(ctx->d_src + i0, rb, rpb, ctx->d_touched + i0, nb, w.fb_id[cur],
                                 w.fb_pos[cur], w.fcell_off[cur], cell_lo, cell_hi, w.feats_out,
                                 w.status, ctx->num_sms, st));
    CK(ctx, cudaEventRecord(ctx->slot_free[s], st));
    ctx->slot_used[s] = true;
  }
  *bytes_out = bytes;
  *hits_out = hits;
  return AGNES_OK;
}

// Row mode: only the requested rows cross the host link.  Touched blocks
// admitted to the cache but not yet loaded are loaded whole first.
//  - Without a feature cache, each distinct requested row crosses once: the
//    tiles' bitmaps of requested ids give every distinct row a staging row in
//    HBM, a loader reads them over the link, and the gather serves every
//    request from staging.
//  - With a feature cache the hot rows, the ones several minibatches request,
//    sit in HBM, and the link carries mostly rows requested once; the gather
//    then reads every row where its block is (cache slot or host memory),
//    so the cached reads overlap the host reads in one pass.
static agnes_status gather_rows_io(agnes_ctx* ctx, int cur, int32_t n, int64_t* bytes_out,
                                   int64_t* hits_out, cudaStream_t st) {
  Workspace& w = ctx->ws;
  const int64_t nfb = ctx->bt.n_feat_blocks;
  const int64_t rpb = ctx->bt.rows_per_feat_block;
  const int64_t rb = ctx->row_bytes;
  const int64_t blk = rpb * rb;
  const int32_t T = (int32_t)ctx->bt.T;
  const int64_t cells = (int64_t)T * w.H;
  const bool dedup = ctx->fcache_slots == 0;
  int32_t nj = 0;
  int64_t bytes = 0, hits = 0, requested_host = 0;
  for (int32_t i = 0; i < n; ++i) {
    const int32_t b = ctx->h_touched[i];
    const int32_t cs = ctx->fcache_slots ? ctx->cslot_of[(size_t)b] : -1;
    if (cs < 0) {
      requested_host += ctx->h_counts[b];
    } else if (ctx->cresident[(size_t)cs]) {
      hits += 1;
    } else {
      ctx->h_job_blk[nj] = b;
      ctx->h_job_dst[nj] = (unsigned long long)(uintptr_t)(ctx->fcache + (int64_t)cs * blk);
      ++nj;
      ctx->cresident[(size_t)cs] = 1;
      ctx->fcache_loads += 1;
      bytes += feat_block_bytes_of(ctx, b);
    }
  }
  for (int64_t b = 0; b < nfb; ++b) {
    const int32_t cs = ctx->fcache_slots ? ctx->cslot_of[(size_t)b] : -1;
    ctx->h_addr[b] = (cs >= 0 && ctx->cresident[(size_t)cs])
                         ? (unsigned long long)(uintptr_t)(ctx->fcache + (int64_t)cs * blk)
                         : (unsigned long long)(uintptr_t)(ctx->features_dev + b * blk);
  }
  CK(ctx, cudaMemcpyAsync(ctx->d_addr, ctx->h_addr, sizeof(unsigned long long) * (size_t)nfb,
                          cudaMemcpyHostToDevice, st));
  if (nj > 0) {
    CK(ctx, cudaMemcpyAsync(ctx->d_job_blk, ctx->h_job_blk, sizeof(int32_t) * nj,
                            cudaMemcpyHostToDevice, st));
    CK(ctx, cudaMemcpyAsync(ctx->d_job_dst, ctx->h_job_dst, sizeof(unsigned long long) * nj,
                            cudaMemcpyHostToDevice, st));
    CK(ctx, launch_load_feat_blocks(ctx->features_dev, ctx->N * rb, ctx->d_job_blk, ctx->d_job_dst,
                                    nj, blk, ctx->num_sms, st));
  }
  ctx->cache_load_bytes = bytes;
  if (!dedup) {
    CK(ctx, launch_gather_table(ctx->d_addr, rb, rpb, w.fb_id[cur], w.fb_pos[cur],
                                w.fcell_off[cur] + cells, w.feats_out, w.status, ctx->num_sms, st));
    ctx->h_rm[1] = requested_host;  // every request of an uncached block crosses the link
    *bytes_out = bytes + requested_host * rb;
    *hits_out = hits;
    return AGNES_OK;
  }
  // distinct requested rows per tile, and their total (for the staging size)
  CK(ctx, launch_tile_bitmaps(w.fb_id[cur], w.fcell_off[cur], ctx->bt.tile_first, T, w.H,
                              ctx->rm_bitmap, ctx->rm_wpref, ctx->rm_dcnt, w.status, st));
  CK(ctx, (seg_scan<int32_t, int32_t>(ctx->rm_dcnt, 0, ctx->rm_doff, 0, nullptr, T, 1, T, true,
                                      nullptr, w.scan_scratch, w.status, st)));
  int32_t* h_total = (int32_t*)ctx->h_rm;
  CK(ctx, cudaMemcpyAsync(h_total, ctx->rm_doff + T, sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaStreamSynchronize(st));
  const int64_t distinct = *h_total;
  if (distinct > ctx->rm_staging_rows) {
    cudaFree(ctx->rm_staging);
    ctx->rm_staging = nullptr;
    ctx->rm_staging_rows = 0;
    const int64_t rows = distinct + distinct / 8 + 1024;
    CK(ctx, cudaMalloc((void**)&ctx->rm_staging, (size_t)(rows * rb)));
    ctx->rm_staging_rows = rows;
  }
  CK(ctx, cudaMemsetAsync(ctx->d_host_rows, 0, sizeof(unsigned long long), st));
  CK(ctx, launch_load_distinct_rows(ctx->d_addr, rb, rpb, ctx->rm_bitmap, ctx->rm_wpref,
                                    ctx->rm_doff, T, ctx->bt.tile_first, ctx->rm_staging, 0, 0,
                                    ctx->d_host_rows, w.status, ctx->num_sms, st));
  CK(ctx, launch_gather_staged_rows(ctx->rm_staging, rb, w.fb_id[cur], w.fb_pos[cur],
                                    w.fcell_off[cur] + cells, ctx->bt.tile_first,
                                    ctx->bt.chunk_tile, T, ctx->rm_bitmap, ctx->rm_wpref,
                                    ctx->rm_doff, ctx->d_addr, rpb, 0, 0, w.feats_out,
                                    w.status, ctx->num_sms, st));
  // rows read over the link, for the counters (read after the hyperbatch is done)
  CK(ctx, cudaMemcpyAsync(ctx->h_rm + 1, ctx->d_host_rows, sizeof(int64_t),
                          cudaMemcpyDeviceToHost, st));
  *bytes_out = bytes + distinct * rb;
  *hits_out = hits;
  return AGNES_OK;
}

// After a hyperbatch: add its requests to the cumulative counts and re-pick
// the cached blocks -- those whose count exceeds the threshold, hottest
// first, up to the cache's capacity.  Blocks that stay keep their slot and
// rows; newly admitted blocks get a free slot and are loaded the next time a
// hyperbatch touches them.  Feature rows are read-only, so a block that
// leaves the cache needs no write-back.
static void update_feature_cache(agnes_ctx* ctx, int32_t n_touched) {
  for (int32_t i = 0; i < n_touched; ++i) {
    const int32_t b = ctx->h_touched[i];
    ctx->acc[(size_t)b] += ctx->h_counts[b];
  }
  const int64_t C = ctx->fcache_slots;
  if (C == 0) return;
  const int64_t nfb = (int64_t)ctx->acc.size();
  std::vector<int32_t> cand;
  cand.reserve((size_t)nfb);
  for (int64_t b = 0; b < nfb; ++b)
    if (ctx->acc[(size_t)b] > 0 && ctx->acc[(size_t)b] > ctx->fcache_threshold)
      cand.push_back((int32_t)b);
  if ((int64_t)cand.size() > C) {
    std::nth_element(cand.begin(), cand.begin() + C, cand.end(), [&](int32_t x, int32_t y) {
      return ctx->acc[(size_t)x] != ctx->acc[(size_t)y] ? ctx->acc[(size_t)x] > ctx->acc[(size_t)y]
                                                        : x < y;
    });
    cand.resize((size_t)C);
  }
  std::vector<uint8_t> keep((size_t)nfb, 0);
  for (int32_t b : cand) keep[(size_t)b] = 1;
  for (int64_t sl = 0; sl < C; ++sl) {  // release slots of blocks that leave
    const int32_t b = ctx->cblock_of[(size_t)sl];
    if (b >= 0 && !keep[(size_t)b]) {
      ctx->cslot_of[(size_t)b] = -1;
      ctx->cblock_of[(size_t)sl] = -1;
      ctx->cresident[(size_t)sl] = 0;
    }
  }
  int64_t free_sl = 0;
  for (int32_t b : cand) {  // admit the new ones into free slots
    if (ctx->cslot_of[(size_t)b] >= 0) continue;
    while (free_sl < C && ctx->cblock_of[(size_t)free_sl] >= 0) ++free_sl;
    if (free_sl >= C) break;
    ctx->cslot_of[(size_t)b] = (int32_t)free_sl;
    ctx->cblock_of[(size_t)free_sl] = b;
    ctx->cresident[(size_t)free_sl] = 0;
  }
}

// Gather with host-resident features.  The request count of every feature
// block (rows gathered from it, over all minibatches) is read back once; the
// touched blocks are those with a request.  Then block mode or row mode runs
// the gather, and the feature cache (Sec. 3.4 (2)) is re-picked.
static agnes_status gather_streamed(agnes_ctx* ctx, int cur, cudaStream_t st) {
  Workspace& w = ctx->ws;
  const int64_t nfb = ctx->bt.n_feat_blocks;
  CK(ctx, launch_count_requests(w.fcell_off[cur], (int32_t)ctx->bt.T, w.H,
                                ctx->bt.tile_feat_block, ctx->d_counts, nfb, true, w.status, st));
  CK(ctx, cudaMemcpyAsync(ctx->h_counts, ctx->d_counts, sizeof(int32_t) * (size_t)nfb,
                          cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaStreamSynchronize(st));
  int32_t n = 0;
  for (int64_t b = 0; b < nfb; ++b)
    if (ctx->h_counts[b]) ctx->h_touched[n++] = (int32_t)b;
  int64_t bytes = 0, hits = 0;
  const agnes_status rc = ctx->feature_io == AGNES_FEATURE_IO_ROWS
                              ? gather_rows_io(ctx, cur, n, &bytes, &hits, st)
                              : gather_blocks_io(ctx, cur, n, &bytes, &hits, st);
  if (rc != AGNES_OK) return rc;
  ctx->streamed_bytes = bytes;
  ctx->streamed_blocks = n - hits;
  ctx->fcache_hits += hits;
  update_feature_cache(ctx, n);
  return AGNES_OK;
}

// Before hyperbatches 2, 2 + R, 2 + 2R, ... (R = kTopoRepickEvery) with a
// topology cache: waits for the previous hyperbatch, reads back the request
// count of every block run since load, and re-picks the cached runs -- most
// requested first, whole runs, up to the cache's capacity.  Runs that stay
// keep their slots; the blocks of newly admitted runs are copied into free
// slots (loader kernel over the host link) and the slot table is uploaded,
// all on st ahead of the hyperbatch.  Re-picking only every R hyperbatches
// keeps the wait (an idle GPU while the host plans) and the churn rare.
static agnes_status update_topology_cache(agnes_ctx* ctx, cudaStream_t st) {
  agnes_ctx::Topo& tp = ctx->topo;
  const int64_t n = ctx->n_prepared;
  if (!tp.cache || n < 1 || (n - 1) % kTopoRepickEvery != 0) return AGNES_OK;
  const int64_t ns = ctx->bt.n_starts, nb = ctx->bt.n_blocks, C = tp.slots;
  CK(ctx, cudaEventSynchronize(ctx->done));  // also: nothing reads the cache while it changes
  CK(ctx, cudaMemcpyAsync(tp.h_acc, tp.d_acc, sizeof(unsigned long long) * (size_t)ns,
                          cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaStreamSynchronize(st));
  const unsigned long long* acc = tp.h_acc;
  std::vector<int32_t> cand;
  for (int64_t r = 0; r < ns; ++r)
    if (acc[r] > 0) cand.push_back((int32_t)r);
  std::sort(cand.begin(), cand.end(),
            [&](int32_t x, int32_t y) { return acc[x] != acc[y] ? acc[x] > acc[y] : x < y; });
  std::vector<uint8_t> keep((size_t)ns, 0);
  int64_t used = 0;
  for (int32_t r : cand) {
    const int64_t m = tp.start_block[(size_t)r + 1] - tp.start_block[(size_t)r];
    if (used + m > C) continue;  // a run too big for what is left; smaller ones may fit
    keep[(size_t)r] = 1;
    used += m;
  }
  std::vector<int32_t> free_slots;
  for (int64_t sl = 0; sl < C; ++sl) {
    const int32_t b = tp.block_of[(size_t)sl];
    if (b >= 0 && keep[(size_t)tp.run_of[(size_t)b]]) continue;
    if (b >= 0) tp.slot_of[(size_t)b] = -1;
    tp.block_of[(size_t)sl] = -1;
    free_slots.push_back((int32_t)sl);
  }
  int32_t njobs = 0;
  for (int32_t r : cand) {
    if (!keep[(size_t)r]) continue;
    for (int32_t b = tp.start_block[(size_t)r]; b < tp.start_block[(size_t)r + 1]; ++b) {
      if (tp.slot_of[(size_t)b] >= 0) continue;
      if (free_slots.empty()) {  // cannot happen: the kept runs fit in C slots
        set_err(ctx, "topology cache out of slots");
        return AGNES_EKERNEL;
      }
      const int32_t sl = free_slots.back();
      free_slots.pop_back();
      tp.slot_of[(size_t)b] = sl;
      tp.block_of[(size_t)sl] = b;
      tp.h_jobs[njobs++] = make_int2(b, sl);
      tp.loaded_blocks += 1;
      tp.loaded_bytes += sizeof(int32_t) * (tp.e1[(size_t)b] - tp.e0[(size_t)b]);
    }
  }
  if (njobs > 0) {
    CK(ctx, cudaMemcpyAsync(tp.d_jobs, tp.h_jobs, sizeof(int2) * (size_t)njobs,
                            cudaMemcpyHostToDevice, st));
    CK(ctx, launch_load_blocks(tp.dev_view, ctx->bt.blk_e0, ctx->bt.blk_e1, tp.d_jobs, njobs,
                               tp.gbuf, tp.epb, ctx->num_sms, st));
  }
  memcpy(tp.h_slot_stage, tp.slot_of.data(), sizeof(int32_t) * (size_t)nb);
  CK(ctx, cudaMemcpyAsync(tp.d_slot, tp.h_slot_stage, sizeof(int32_t) * (size_t)nb,
                          cudaMemcpyHostToDevice, st));
  return AGNES_OK;
}

// Enqueues one hyperbatch on st whose targets are already in w.nodes and whose
// sampling key is in w.key: the bucketing of the targets, K hops of sampling
// and dedup, the feature gather, the statistics and the size read-back.
// mark_flags is cudaEventRecordExternal while the sequence is being captured,
// so the phase events become event-record nodes of the graph; *n_marks gets
// the number of phase events recorded.
static agnes_status enqueue_hyperbatch(agnes_ctx* ctx, const int32_t* fanouts, int32_t K,
                                       const int64_t* cap, int ring, unsigned mark_flags,
                                       cudaStream_t st, int* n_marks) {
  agnes_status rc = AGNES_OK;
  Workspace& w = ctx->ws;
  const int32_t H = w.H, B = w.B;
  const int32_t T = (int32_t)ctx->bt.T;
  const int64_t cells = (int64_t)T * H;
  const int nsm = ctx->num_sms;
  int ph = 0;
  auto mark = [&]() {
    if (ctx->profiling) cudaEventRecordWithFlags(ctx->ev[ring][ph++], st, mark_flags);
  };

  mark();
  CK(ctx, cudaMemsetAsync(w.status, 0, sizeof(int32_t), st));
  CK(ctx, cudaMemsetAsync(w.fcnt, 0, sizeof(int32_t) * cells, st));
  CK(ctx, cudaMemsetAsync(w.adj_flags, 0, (size_t)K * ctx->bt.n_blocks, st));
  CK(ctx, cudaMemsetAsync(w.feat_flags, 0, (size_t)ctx->bt.n_feat_blocks, st));
  CK(ctx, cudaMemsetAsync(w.stats, 0, sizeof(int64_t) * (K + 1), st));
  fill_i32_kernel<<<(H + 255) / 256, 256, 0, st>>>(w.nsz, H, B);
  CK(ctx, cudaGetLastError());
  CK(ctx, launch_bucket_targets(w.nodes, w.capK, H, B, (int32_t)ctx->N, ctx->bt.tile_first,
                                ctx->bt.chunk_tile, T, w.fcnt, w.fcell_off[0], w.tmp_id, w.tmp_pos,
                                w.fb_id[0], w.fb_pos[0], w.scan_scratch, w.status, nsm, st));
  int cur = 0;
  for (int h = 0; h < K; ++h) {
    mark();
    HopArgs a;
    a.offsets = ctx->offsets;
    a.offsets_bits = ctx->offsets_bits;
    a.indices = ctx->indices;
    a.N = (int32_t)ctx->N;
    a.tile_first = ctx->bt.tile_first;
    a.chunk_tile = ctx->bt.chunk_tile;
    a.T = T;
    a.H = H;
    a.capK = w.capK;
    a.cap_prev = cap[h];
    a.ecap = cap[h] * fanouts[h];
    a.k = fanouts[h];
    a.hop = h + 1;
    a.key = w.key;
    a.status = w.status;
    int32_t* nsz_prev = w.nsz + (int64_t)h * H;
    int32_t* ecnt = w.ecnt + (int64_t)h * H;
    CK(ctx, launch_sample_count(a, w.fb_id[cur], w.fb_pos[cur], w.fcell_off[cur], w.cnt, nsm, st));
    CK(ctx, (seg_scan<int32_t, int64_t>(w.cnt, cap[h], w.indptr[h], cap[h] + 1, nsz_prev, 0, H,
                                         cap[h], true, ecnt, w.scan_scratch, w.status, st)));
    mark();
    CK(ctx, cudaMemsetAsync(w.scnt, 0, sizeof(int32_t) * cells, st));
    if (ctx->topo.on) {
      rc = fill_streamed(ctx, a, cur, h, st);
      if (rc != AGNES_OK) return rc;
    } else {
      FillRange r;
      r.cell_lo = 0;
      r.cell_hi = cells;
      const agnes_ctx::Topo& tp = ctx->topo;
      if (tp.cache) {  // requests per block run, then cached blocks from HBM, others in place
        CK(ctx, launch_count_cache_requests(w.fcell_off[cur], T, H, ctx->bt.tile_adj_start,
                                            ctx->bt.tile_adj_block, tp.d_slot, tp.d_acc,
                                            tp.d_cached, w.status, st));
        r.tile_adj_block = ctx->bt.tile_adj_block;
        r.blk_slot = tp.d_slot;
        r.blk_e0 = ctx->bt.blk_e0;
        r.gbuf = tp.gbuf;
        r.epb = tp.epb;
        r.bb = ctx->adj_block_bytes;
        r.in_place_fallback = true;
      }
      CK(ctx, launch_sample_fill(a, w.fb_id[cur], w.fb_pos[cur], w.fcell_off[cur], w.indptr[h],
                                 w.nbr, w.scnt, w.scell, w.srank, r, nsm, st));
    }
    mark();
    DedupBufs d;
    d.nbr = w.nbr;
    d.ecnt = ecnt;
    d.scell = w.scell;
    d.srank = w.srank;
    d.scnt = w.scnt;
    d.soff = w.soff;
    d.sb = w.sb;
    d.tmp = w.tmp;
    d.big_list = w.big_list;
    d.big_n = w.big_n;
    d.fb_id = w.fb_id[cur];
    d.fb_pos = w.fb_pos[cur];
    d.fcell_off = w.fcell_off[cur];
    d.newcnt = w.newcnt;
    d.newbase = w.newbase;
    d.nfcnt = w.nfcnt;
    d.nfcell_off = w.fcell_off[1 - cur];
    d.nfb_id = w.fb_id[1 - cur];
    d.nfb_pos = w.fb_pos[1 - cur];
    d.nsz_prev = nsz_prev;
    d.nsz_next = w.nsz + (int64_t)(h + 1) * H;
    d.srcsz = w.srcsz + (int64_t)h * H;
    d.noutbase = w.noutbase;
    d.frontier_sampled = ctx->frontier_mode == AGNES_FRONTIER_SAMPLED && h + 1 < K;
    d.nodes = w.nodes;
    d.col = w.col[h];
    d.tile_adj_block = ctx->bt.tile_adj_block;
    d.adj_flags = w.adj_flags + (int64_t)h * ctx->bt.n_blocks;
    d.scan_scratch = w.scan_scratch;
    CK(ctx, launch_dedup(a, d, nsm, st));
    cur = 1 - cur;
  }
  // feature blocks touched by the hyperbatch (stats; also the streaming list)
  CK(ctx, launch_mark_count(w.fcell_off[cur], T, H, ctx->bt.tile_feat_block, w.feat_flags,
                            ctx->bt.n_feat_blocks, w.stats + K, w.status, st));
  mark();
  if (ctx->features_on_host) {
    rc = gather_streamed(ctx, cur, st);
    if (rc != AGNES_OK) return rc;
  } else {
    CK(ctx, launch_gather(ctx->features, ctx->row_bytes, w.fb_id[cur], w.fb_pos[cur],
                          w.fcell_off[cur] + cells, w.feats_out, w.status, nsm, st));
  }
  mark();
  for (int h = 0; h < K; ++h)
    CK(ctx, launch_mark_count(nullptr, T, H, nullptr, w.adj_flags + (int64_t)h * ctx->bt.n_blocks,
                              ctx->bt.n_blocks, w.stats + h, w.status, st));
  const Back b = back_of(w);
  CK(ctx, cudaMemcpyAsync(b.status, w.status, sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaMemcpyAsync(b.nsz, w.nsz, sizeof(int32_t) * (K + 1) * H, cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaMemcpyAsync(b.ecnt, w.ecnt, sizeof(int32_t) * K * H, cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaMemcpyAsync(b.srcsz, w.srcsz, sizeof(int32_t) * K * H, cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaMemcpyAsync(b.stats, w.stats, sizeof(int64_t) * (K + 1), cudaMemcpyDeviceToHost, st));
  if (ctx->topo.cache)
    CK(ctx, cudaMemcpyAsync(ctx->topo.h_cached, ctx->topo.d_cached, sizeof(unsigned long long),
                            cudaMemcpyDeviceToHost, st));
  *n_marks = ph;
  return AGNES_OK;
}


// Whether work enqueued on st is being captured (by the caller's own graph
// capture); an unknown state counts as captured, so the sequence is enqueued
// as it is.
static bool stream_capturing(cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) {
    cudaGetLastError();
    return true;
  }
  return cs != cudaStreamCaptureStatusNone;
}

// Turns every kernel-to-kernel edge of the captured sequence into a
// programmatic one from the programmatic port: the kernels trigger nothing
// early, so the next kernel is launched as soon as every block of its
// predecessor has exited, and its blocks wait at their first statement
// (grid_dep_wait) for the predecessor's writes to become visible; the launch
// overlaps the predecessor's completion instead of following it.  (Launching
// once all predecessor blocks had merely started was measured slower: the
// waiting blocks took SM slots from the running kernel's tail.)  Edges
// touching other nodes (memsets, copies, event records) keep full
// serialisation.
static cudaError_t make_programmatic(cudaGraph_t graph, int64_t* converted) {
  size_t n = 0;
  cudaError_t e = cudaGraphGetEdges(graph, nullptr, nullptr, nullptr, &n);
  if (e != cudaSuccess || n == 0) return e;
  std::vector<cudaGraphNode_t> from(n), to(n);
  std::vector<cudaGraphEdgeData> data(n);
  e = cudaGraphGetEdges(graph, from.data(), to.data(), data.data(), &n);
  if (e != cudaSuccess) return e;
  for (size_t i = 0; i < n; ++i) {
    cudaGraphNodeType tf, tt;
    if ((e = cudaGraphNodeGetType(from[i], &tf)) != cudaSuccess) return e;
    if ((e = cudaGraphNodeGetType(to[i], &tt)) != cudaSuccess) return e;
    if (tf != cudaGraphNodeTypeKernel || tt != cudaGraphNodeTypeKernel) continue;
    if (data[i].type != cudaGraphDependencyTypeDefault || data[i].from_port != 0) continue;
    if ((e = cudaGraphRemoveDependencies(graph, &from[i], &to[i], &data[i], 1)) != cudaSuccess)
      return e;
    cudaGraphEdgeData p;
    memset(&p, 0, sizeof(p));
    p.from_port = cudaGraphKernelNodePortProgrammatic;
    p.type = cudaGraphDependencyTypeProgrammatic;
    if ((e = cudaGraphAddDependencies(graph, &from[i], &to[i], &p, 1)) != cudaSuccess) return e;
    *converted += 1;
  }
  return cudaSuccess;
}

// The resident path as one graph launch.  The launch sequence is captured on
// a private stream the first time a hyperbatch shape (H, B, fanouts, frontier
// mode, profiling, workspace) is seen, and replayed for every later hyperbatch
// of that shape: everything that varies between them (the targets, the seed,
// the minibatch ids) is in device memory by then.  With profiling on, the
// captured phase-event nodes are pointed at this prepare's ring slot.
static agnes_status launch_graphed(agnes_ctx* ctx, const int32_t* fanouts, int32_t K,
                                   const int64_t* cap, int ring, cudaStream_t st,
                                   int* n_marks) {
  agnes_ctx::LaunchGraph& g = ctx->lg;
  const Workspace& w = ctx->ws;
  bool same = g.exec && g.H == w.H && g.B == w.B && g.K == K &&
              g.frontier_mode == ctx->frontier_mode && g.profiling == ctx->profiling &&
              g.ws_gen == ctx->ws_gen && g.built_mode == g.mode;
  for (int h = 0; same && h < K; ++h) same = g.fan[h] == fanouts[h];
  if (!same) {
    drop_launch_graph(&g);
    if (!g.cap) CK(ctx, cudaStreamCreateWithFlags(&g.cap, cudaStreamNonBlocking));
    CK(ctx, cudaStreamBeginCapture(g.cap, cudaStreamCaptureModeRelaxed));
    int nm = 0;
    const agnes_status rc =
        enqueue_hyperbatch(ctx, fanouts, K, cap, ring, cudaEventRecordExternal, g.cap, &nm);
    cudaGraph_t graph = nullptr;
    const cudaError_t e = cudaStreamEndCapture(g.cap, &graph);
    if (rc != AGNES_OK || e != cudaSuccess) {
      if (graph) cudaGraphDestroy(graph);
      cudaGetLastError();
      if (rc != AGNES_OK) return rc;
      set_err(ctx, "capturing the launch sequence failed: %s", cudaGetErrorString(e));
      return AGNES_ECUDA;
    }
    g.graph = graph;
    g.programmatic_edges = 0;
    if (g.mode == AGNES_LAUNCH_GRAPH_PDL) CK(ctx, make_programmatic(graph, &g.programmatic_edges));
    CK(ctx, cudaGraphInstantiate(&g.exec, graph, 0));
    if (ctx->profiling) {
      size_t n = 0;
      CK(ctx, cudaGraphGetNodes(graph, nullptr, &n));
      std::vector<cudaGraphNode_t> nodes(n);
      CK(ctx, cudaGraphGetNodes(graph, nodes.data(), &n));
      for (int i = 0; i < nm; ++i) g.phase_node[i] = nullptr;
      for (cudaGraphNode_t nd : nodes) {
        cudaGraphNodeType t;
        CK(ctx, cudaGraphNodeGetType(nd, &t));
        if (t != cudaGraphNodeTypeEventRecord) continue;
        cudaEvent_t ev = nullptr;
        CK(ctx, cudaGraphEventRecordNodeGetEvent(nd, &ev));
        for (int i = 0; i < nm; ++i)
          if (ctx->ev[ring][i] == ev) g.phase_node[i] = nd;
      }
      for (int i = 0; i < nm; ++i) {
        if (!g.phase_node[i]) {
          drop_launch_graph(&g);
          set_err(ctx, "phase event %d is missing from the captured launch sequence", i);
          return AGNES_ECUDA;
        }
      }
    }
    g.n_marks = nm;
    g.H = w.H;
    g.B = w.B;
    g.K = K;
    for (int h = 0; h < K; ++h) g.fan[h] = fanouts[h];
    g.frontier_mode = ctx->frontier_mode;
    g.built_mode = g.mode;
    g.profiling = ctx->profiling;
    g.ws_gen = ctx->ws_gen;
    g.captures += 1;
  }
  if (g.profiling)
    for (int i = 0; i < g.n_marks; ++i)
      CK(ctx, cudaGraphExecEventRecordNodeSetEvent(g.exec, g.phase_node[i], ctx->ev[ring][i]));
  CK(ctx, cudaGraphLaunch(g.exec, st));
  g.launches += 1;
  *n_marks = g.n_marks;
  return AGNES_OK;
}

agnes_status agnes_prepare_hyperbatch(agnes_ctx* ctx, const int32_t* targets, int32_t H,
                                      int32_t B, const int32_t* fanouts, int32_t K,
                                      uint64_t seed, uint64_t first_minibatch_id,
                                      void* cuda_stream) {
  if (!ctx) {
    set_err(nullptr, "ctx is NULL");
    return AGNES_EINVAL;
  }
  if (!targets || !fanouts) {
    set_err(ctx, "targets and fanouts must be non-NULL");
    return AGNES_EINVAL;
  }
  if (H < 1 || H > 65535 || B < 1 || K < 1 || K > AGNES_MAX_HOPS) {
    set_err(ctx, "need 1 <= H <= 65535, B >= 1, 1 <= K <= %d", AGNES_MAX_HOPS);
    return AGNES_EINVAL;
  }
  if (B > ctx->N) {
    set_err(ctx, "B = %d distinct targets exceed N = %lld", B, (long long)ctx->N);
    return AGNES_EINVAL;
  }
  int64_t cap[AGNES_MAX_HOPS + 1];
  cap[0] = B;
  for (int h = 0; h < K; ++h) {
    if (fanouts[h] < 1 || fanouts[h] > AGNES_MAX_FANOUT) {
      set_err(ctx, "fanouts[%d] = %d outside [1, %d]", h, fanouts[h], AGNES_MAX_FANOUT);
      return AGNES_EINVAL;
    }
    const int64_t grown = cap[h] * (1 + (int64_t)fanouts[h]);
    cap[h + 1] = grown < ctx->N ? grown : ctx->N;
  }
  const int64_t lim = ((int64_t)1 << 31) - 1;
  for (int h = 0; h < K; ++h) {
    if ((int64_t)H * cap[h] * fanouts[h] > lim) {
      set_err(ctx, "H x edge capacity of hop %d exceeds 2^31", h + 1);
      return AGNES_ERANGE;
    }
  }
  if ((int64_t)H * cap[K] > lim) {
    set_err(ctx, "H x node capacity (%lld) exceeds 2^31", (long long)(H * cap[K]));
    return AGNES_ERANGE;
  }
  if (cudaSetDevice(ctx->device) != cudaSuccess) {
    cudaGetLastError();
    set_err(ctx, "cudaSetDevice failed");
    return AGNES_ECUDA;
  }
  agnes_status rc = ensure_workspace(ctx, H, B, fanouts, K, cap);
  if (rc != AGNES_OK) return rc;
  Workspace& w = ctx->ws;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  ctx->prepared = false;
  ctx->synced = false;
  if (ctx->profiling && !ctx->ev_created) {
    for (int r = 0; r < kEventRing; ++r)
      for (int i = 0; i <= kMaxPhases; ++i) CK(ctx, cudaEventCreate(&ctx->ev[r][i]));
    ctx->ev_created = true;
  }
  const int ring = (int)(ctx->n_prepared % kEventRing);
  ctx->n_phases[ring] = 0;
  // a prepare on another stream than the last one still runs after it: both
  // use the ctx's buffers (a caller's own capture orders its replays itself)
  const bool capturing = stream_capturing(st);
  if (ctx->n_prepared > 0 && !capturing) CK(ctx, cudaStreamWaitEvent(st, ctx->done, 0));
  if (!capturing) {
    rc = update_topology_cache(ctx, st);
    if (rc != AGNES_OK) return rc;
  }
  CK(ctx, cudaMemcpy2DAsync(w.nodes, sizeof(int32_t) * w.capK, targets, sizeof(int32_t) * B,
                            sizeof(int32_t) * B, H, cudaMemcpyDefault, st));
  CK(ctx, launch_set_key(w.key, seed, first_minibatch_id, st));
  int n_marks = 0;
  const bool resident = !ctx->features_on_host && !ctx->topo.on;
  if (resident && ctx->lg.mode != AGNES_LAUNCH_DIRECT && !capturing)
    rc = launch_graphed(ctx, fanouts, K, cap, ring, st, &n_marks);
  else
    rc = enqueue_hyperbatch(ctx, fanouts, K, cap, ring, cudaEventRecordDefault, st, &n_marks);
  if (rc != AGNES_OK) return rc;
  // inside a caller's capture nothing has run yet: the caller orders its
  // replays, and there are no phase times to read
  if (!capturing) CK(ctx, cudaEventRecord(ctx->done, st));
  ctx->n_phases[ring] = ctx->profiling && !capturing ? n_marks - 1 : 0;
  ctx->n_prepared += 1;
  ctx->cur = K & 1;  // the frontier buffers swap once per hop
  ctx->prepared = true;
  return AGNES_OK;
}


agnes_status agnes_fetch_minibatch(agnes_ctx* ctx, int32_t j, agnes_minibatch_view* out) {
  if (!ctx || !out) {
    set_err(ctx, "ctx and out must be non-NULL");
    return AGNES_EINVAL;
  }
  agnes_status rc = wait_prepared(ctx);
  if (rc != AGNES_OK) return rc;
  Workspace& w = ctx->ws;
  if (j < 0 || j >= w.H) {
    set_err(ctx, "minibatch %d outside [0, %d)", j, w.H);
    return AGNES_EINVAL;
  }
  const Back b = back_of(w);
  memset(out, 0, sizeof(*out));
  out->K = w.K;
  for (int h = 0; h < w.K; ++h) {
    out->num_dst[h] = b.nsz[(size_t)h * w.H + j];
    out->num_src[h] = b.srcsz[(size_t)h * w.H + j];
    out->num_edges[h] = b.ecnt[(size_t)h * w.H + j];
    out->indptr[h] = w.indptr[h] + (int64_t)j * (w.cap[h] + 1);
    out->col[h] = w.col[h] + (int64_t)j * w.cap[h] * w.fan[h];
  }
  out->nodes = w.nodes + (int64_t)j * w.capK;
  out->num_nodes = b.nsz[(size_t)w.K * w.H + j];
  out->feats = (const char*)w.feats_out + (int64_t)j * w.capK * ctx->row_bytes;
  out->feat_dtype = ctx->feat_dtype;
  out->feat_dim = ctx->feat_dim;
  return AGNES_OK;
}

agnes_status agnes_set_frontier_mode(agnes_ctx* ctx, int32_t mode) {
  if (!ctx) return AGNES_EINVAL;
  if (mode != AGNES_FRONTIER_SRC && mode != AGNES_FRONTIER_SAMPLED) {
    set_err(ctx, "frontier mode must be AGNES_FRONTIER_SRC or AGNES_FRONTIER_SAMPLED");
    return AGNES_EINVAL;
  }
  ctx->frontier_mode = mode;
  return AGNES_OK;
}

agnes_status agnes_set_launch_mode(agnes_ctx* ctx, int32_t mode) {
  if (!ctx) return AGNES_EINVAL;
  if (mode != AGNES_LAUNCH_DIRECT && mode != AGNES_LAUNCH_GRAPH && mode != AGNES_LAUNCH_GRAPH_PDL) {
    set_err(ctx, "launch mode must be AGNES_LAUNCH_DIRECT, _GRAPH or _GRAPH_PDL");
    return AGNES_EINVAL;
  }
  ctx->lg.mode = mode;
  return AGNES_OK;
}

agnes_status agnes_fetch_hyperbatch(agnes_ctx* ctx, agnes_hyperbatch_view* out) {
  if (!ctx || !out) {
    set_err(ctx, "ctx and out must be non-NULL");
    return AGNES_EINVAL;
  }
  agnes_status rc = wait_prepared(ctx);
  if (rc != AGNES_OK) return rc;
  Workspace& w = ctx->ws;
  const Back b = back_of(w);
  memset(out, 0, sizeof(*out));
  out->K = w.K;
  out->H = w.H;
  for (int h = 0; h < w.K; ++h) {
    out->indptr[h] = w.indptr[h];
    out->indptr_stride[h] = w.cap[h] + 1;
    out->col[h] = w.col[h];
    out->col_stride[h] = w.cap[h] * w.fan[h];
  }
  out->nodes = w.nodes;
  out->nodes_stride = w.capK;
  out->feats = w.feats_out;
  out->feats_stride_rows = w.capK;
  out->feat_dtype = ctx->feat_dtype;
  out->feat_dim = ctx->feat_dim;
  out->node_size = b.nsz;
  out->edges = b.ecnt;
  out->src_size = b.srcsz;
  return AGNES_OK;
}

agnes_status agnes_hyperbatch_stats(agnes_ctx* ctx, int64_t* out) {
  if (!ctx || !out) {
    set_err(ctx, "ctx and out must be non-NULL");
    return AGNES_EINVAL;
  }
  agnes_status rc = wait_prepared(ctx);
  if (rc != AGNES_OK) return rc;
  const Back b = back_of(ctx->ws);
  for (int h = 0; h <= ctx->ws.K; ++h) out[h] = b.stats[h];
  return AGNES_OK;
}

agnes_status agnes_hyperbatch_counters(agnes_ctx* ctx, agnes_counters* out) {
  if (!ctx || !out) {
    set_err(ctx, "ctx and out must be non-NULL");
    return AGNES_EINVAL;
  }
  agnes_status rc = wait_prepared(ctx);
  if (rc != AGNES_OK) return rc;
  Workspace& w = ctx->ws;
  const Back b = back_of(w);
  memset(out, 0, sizeof(*out));
  out->K = w.K;
  for (int h = 0; h < w.K; ++h)
    for (int j = 0; j < w.H; ++j) {
      out->frontier[h] += b.nsz[(size_t)h * w.H + j];
      out->edges[h] += b.ecnt[(size_t)h * w.H + j];
    }
  for (int j = 0; j < w.H; ++j) out->rows += b.nsz[(size_t)w.K * w.H + j];
  out->row_bytes = ctx->row_bytes;
  cudaSetDevice(ctx->device);
  unsigned long long distinct = 0;
  CK(ctx, cudaMemset(w.distinct, 0, sizeof(unsigned long long)));
  CK(ctx, launch_distinct_rows(w.fb_id[ctx->cur], w.fcell_off[ctx->cur], ctx->bt.tile_first,
                               (int32_t)ctx->bt.T, w.H, w.distinct, nullptr));
  CK(ctx, cudaMemcpy(&distinct, w.distinct, sizeof(distinct), cudaMemcpyDeviceToHost));
  out->distinct_rows = (int64_t)distinct;
  out->streamed_bytes = !ctx->features_on_host ? 0
                        : ctx->feature_io == AGNES_FEATURE_IO_ROWS
                            ? ctx->cache_load_bytes + ctx->h_rm[1] * ctx->row_bytes
                            : ctx->streamed_bytes;
  out->streamed_blocks = ctx->features_on_host ? ctx->streamed_blocks : 0;
  out->topo_loaded_blocks = ctx->topo.loaded_blocks;
  out->topo_loaded_bytes = ctx->topo.loaded_bytes;
  out->topo_hit_blocks = ctx->topo.hits;
  out->topo_cached_requests = ctx->topo.cache ? (int64_t)*ctx->topo.h_cached : 0;
  out->topo_waves = ctx->topo.waves;
  out->fcache_hit_blocks = ctx->fcache_hits;
  out->fcache_loaded_blocks = ctx->fcache_loads;
  out->graph_captures = ctx->lg.captures;
  out->graph_launches = ctx->lg.launches;
  out->graph_programmatic_edges = ctx->lg.programmatic_edges;
  return AGNES_OK;
}

agnes_status agnes_get_graph_info(agnes_ctx* ctx, agnes_graph_info* out) {
  if (!ctx || !out) {
    set_err(ctx, "ctx and out must be non-NULL");
    return AGNES_EINVAL;
  }
  out->num_nodes = ctx->N;
  out->num_edges = ctx->E;
  out->adj_blocks = ctx->bt.n_blocks;
  out->adj_block_starts = ctx->bt.n_starts;
  out->feat_blocks = ctx->bt.n_feat_blocks;
  out->feat_rows_per_block = ctx->bt.rows_per_feat_block;
  out->tiles = ctx->bt.T;
  out->row_bytes = ctx->row_bytes;
  return AGNES_OK;
}

agnes_status agnes_copy_adj_blocks(agnes_ctx* ctx, int32_t* start_node, int32_t* start_block,
                                   int64_t cap) {
  if (!ctx || !start_node || !start_block || cap < 0) {
    set_err(ctx, "invalid arguments");
    return AGNES_EINVAL;
  }
  const int64_t n = cap < ctx->bt.n_starts ? cap : ctx->bt.n_starts;
  cudaSetDevice(ctx->device);
  CK(ctx, cudaMemcpy(start_node, ctx->bt.start_node, sizeof(int32_t) * n, cudaMemcpyDeviceToHost));
  CK(ctx, cudaMemcpy(start_block, ctx->bt.start_block, sizeof(int32_t) * n,
                     cudaMemcpyDeviceToHost));
  return AGNES_OK;
}

agnes_status agnes_set_profiling(agnes_ctx* ctx, int32_t enable) {
  if (!ctx) return AGNES_EINVAL;
  ctx->profiling = enable != 0;
  return AGNES_OK;
}

agnes_status agnes_phase_times(agnes_ctx* ctx, int32_t ago, float* ms, int32_t n,
                               int32_t* n_out) {
  if (!ctx || (!ms && n > 0) || !n_out || ago < 0 || ago >= kEventRing) {
    set_err(ctx, "invalid arguments");
    return AGNES_EINVAL;
  }
  *n_out = 0;
  agnes_status rc = wait_prepared(ctx);
  if (rc != AGNES_OK) return rc;
  if (ago >= ctx->n_prepared) {
    set_err(ctx, "only %lld hyperbatches prepared", (long long)ctx->n_prepared);
    return AGNES_EINVAL;
  }
  const int ring = (int)((ctx->n_prepared - 1 - ago) % kEventRing);
  const int cnt = ctx->n_phases[ring] < n ? ctx->n_phases[ring] : n;
  for (int i = 0; i < cnt; ++i)
    CK(ctx, cudaEventElapsedTime(&ms[i], ctx->ev[ring][i], ctx->ev[ring][i + 1]));
  *n_out = cnt;
  return AGNES_OK;
}

}  // extern "C"
