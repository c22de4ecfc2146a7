// ctx.h -- the library context behind the C ABI's opaque agnes_ctx handle,
// shared by the host-side translation units:
//   api.cu            the C ABI entry points: graph load, views, statistics
//   prepare.cu        one hyperbatch: workspace, launch sequence, CUDA graph
//   host_features.cu  features in pinned host memory: block / row I/O, cache
//   topology.cu       topology in pinned host memory: graph buffer, cache
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "../../include/agnes.h"
#include "common.cuh"
#include "internal.h"

namespace agnes {

constexpr int kMaxPhases = 2 + 3 * AGNES_MAX_HOPS;
constexpr int kEventRing = 64;  // prepares whose phase times stay readable
// Streaming of host-resident features: a ring of staging slots in HBM, each
// holding a batch of up to kStreamBatchBlocks touched feature blocks.
constexpr int kStreamSlots = 4;
constexpr int kStreamBatchBlocks = 64;
// Row I/O of host-resident features: the distinct rows are loaded in this many
// tile ranges, each range's gather starting once its rows are in.
constexpr int kRowChunks = 8;
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
  int32_t* hset = nullptr;     // fanouts above kWideMax: the sampler's per-warp hash sets
  int64_t hset_elems = 0;
  int32_t* q_cells = nullptr;  // default frontier's dedup queue (internal.h, DedupBufs)
  int32_t* q_cnt = nullptr;
  int32_t* q_off = nullptr;
  int32_t* q_dense = nullptr;
  int32_t* q_next = nullptr;
  int32_t q_chunks_cap = 0;
  int32_t* big_n = nullptr;
  int32_t* tmp_id = nullptr;
  int32_t* tmp_pos = nullptr;
  int32_t* cnt = nullptr;
  int64_t* fbd = nullptr;  // 2 per frontier entry: (first edge, degree)
  uint64_t* flat_scratch = nullptr;  // single-pass scans of the cell counts (zero between scans)
  int64_t flat_elems = 0;
  void* feats_out = nullptr;
  uint8_t* adj_flags = nullptr;
  uint8_t* feat_flags = nullptr;
  int64_t* stats = nullptr;  // K+1
  int64_t* scan_scratch = nullptr;
  int64_t* side_scratch = nullptr;  // scans on the side stream
  int32_t* status = nullptr;
  unsigned long long* distinct = nullptr;
  uint64_t* key = nullptr;  // sampling key {seed, first minibatch id}

  // pinned host readback: [status][nsz (K+1)H][ecnt KH][srcsz KH] then int64 stats (K+1)
  void* h_back = nullptr;
  size_t h_back_bytes = 0;
};

// Host view of the readback buffer.
struct Back {
  int32_t* status;
  int32_t* nsz;
  int32_t* ecnt;
  int32_t* srcsz;
  int64_t* stats;
};

inline Back back_of(Workspace& w) {
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

}  // namespace agnes

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
  agnes::BlockTables bt;

  agnes::Workspace ws;
  bool prepared = false;
  bool synced = false;
  int cur = 0;  // which frontier buffer holds the final bucket
  cudaEvent_t done = nullptr;

  int32_t profiling = AGNES_PROFILE_OFF;
  int64_t n_prepared = 0;                  // prepares issued so far
  int n_phases[agnes::kEventRing] = {0};          // per ring slot; 0 = not profiled
  cudaEvent_t ev[agnes::kEventRing][agnes::kMaxPhases + 1] = {{nullptr}};
  bool ev_created = false;
  uint64_t ws_gen = 0;  // bumped whenever the workspace is reallocated
  // side stream of a hyperbatch: each hop's new-id scan and col fix-up run on
  // it (forked after the cells are resolved; the compaction waits for the
  // scan through aux_ready; joined before the next hop's sampling), and the
  // touched-block statistics (forked before the last compaction, joined
  // before the size read-back)
  cudaStream_t aux = nullptr;
  cudaEvent_t aux_fork = nullptr, aux_join = nullptr, aux_ready = nullptr;

  // The resident path's launch sequence, captured once per hyperbatch shape
  // and replayed as one CUDA graph launch (agnes_set_launch_mode).
  struct LaunchGraph {
    int32_t mode = AGNES_LAUNCH_GRAPH_PDL;
    cudaStream_t cap = nullptr;  // private stream the sequence is captured on
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    // what the capture depends on
    int32_t H = 0, B = 0, K = 0, fan[AGNES_MAX_HOPS] = {0}, frontier_mode = 0, built_mode = 0;
    int32_t profiling = AGNES_PROFILE_OFF;
    uint64_t ws_gen = 0;
    // phase-event nodes, re-pointed at each launch's ring slot
    cudaGraphNode_t phase_node[agnes::kMaxPhases + 1] = {nullptr};
    int n_marks = 0;
    int64_t captures = 0, launches = 0, programmatic_edges = 0;
  } lg;

  // Hyperbatches in flight (agnes_set_pipeline_depth): with a depth of d > 1
  // the ctx keeps d - 1 more sets of the per-hyperbatch state -- workspace,
  // launch graph, completion and side-stream events, side stream, its own
  // internal stream and the fetch state -- and rotates them with the active
  // set at every prepare, so consecutive hyperbatches use the sets in turn
  // and run on their internal streams, overlapping.  The active set (the
  // fields above and pipe_st) always belongs to the last prepare; spares[0]
  // to the oldest hyperbatch still held, spares[d - 2] to the one before the
  // last.
  int32_t pipe_depth = 1;
  cudaStream_t pipe_st = nullptr;  // the active set's internal stream (depth > 1)
  cudaEvent_t pipe_in = nullptr;   // orders an internal stream after the caller's
  struct Spare {
    agnes::Workspace ws;
    LaunchGraph lg;
    uint64_t ws_gen = 0;
    cudaEvent_t done = nullptr, aux_fork = nullptr, aux_join = nullptr, aux_ready = nullptr;
    cudaStream_t aux = nullptr;
    cudaStream_t pipe_st = nullptr;
    int cur = 0;
    bool prepared = false, synced = false;
  } spares[AGNES_MAX_PIPELINE_DEPTH - 1];

  // streaming of host-resident features (features_on_host)
  cudaStream_t copy_stream = nullptr;
  char* slots = nullptr;
  int64_t slot_bytes = 0;
  cudaEvent_t slot_copied[agnes::kStreamSlots] = {nullptr};
  cudaEvent_t slot_free[agnes::kStreamSlots] = {nullptr};
  bool slot_used[agnes::kStreamSlots] = {false};
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
  cudaEvent_t rows_loaded[agnes::kRowChunks] = {nullptr};  // row I/O: per tile range
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

// Sets the ctx's (or, without a ctx, the thread's) last error message.
#define set_err ctx_set_error

// Returns AGNES_ECUDA (AGNES_ENOMEM for an allocation) from the calling
// function when a CUDA call fails, with the call in the error message.
#define CK(ctx, call)                                                            \
  do {                                                                           \
    cudaError_t e_ = (call);                                                     \
    if (e_ != cudaSuccess) {                                                     \
      set_err(ctx, "%s failed: %s", #call, cudaGetErrorString(e_));              \
      return e_ == cudaErrorMemoryAllocation ? AGNES_ENOMEM : AGNES_ECUDA;       \
    }                                                                            \
  } while (0)

// prepare.cu
void free_workspace(agnes::Workspace* w);
void drop_launch_graph(agnes_ctx::LaunchGraph* g);
// Swaps the active per-hyperbatch state with spare set o.
void swap_hyperbatch_state(agnes_ctx* ctx, agnes_ctx::Spare& o);
// Before a prepare at depth d > 1: the oldest set (spares[0]) becomes the
// active one and the active one the newest spare (spares[d - 2]).
void rotate_hyperbatch_state(agnes_ctx* ctx);
// Creates the events and streams of spares[0 .. depth - 2] (once); frees
// every spare set.
agnes_status make_spare_state(agnes_ctx* ctx, int32_t depth);
void free_spare_state(agnes_ctx* ctx);

// host_features.cu
agnes_status setup_streaming(agnes_ctx* ctx, const agnes_graph_desc* d, cudaStream_t st);
agnes_status gather_streamed(agnes_ctx* ctx, int cur, cudaStream_t st);

// topology.cu
agnes_status setup_topology(agnes_ctx* ctx, const agnes_graph_desc* d, cudaStream_t st);
agnes_status setup_topology_cache(agnes_ctx* ctx, const agnes_graph_desc* d, cudaStream_t st);
agnes_status fill_streamed(agnes_ctx* ctx, const agnes::HopArgs& a, int cur, int h,
                           cudaStream_t st);
agnes_status update_topology_cache(agnes_ctx* ctx, cudaStream_t st);
