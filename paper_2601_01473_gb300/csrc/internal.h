// internal.h -- host-side launchers shared between the libagnes translation
// units.  Not part of the public ABI (include/agnes.h is).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace agnes {

// ---- scan.cu ---------------------------------------------------------------
// CTAs of `threads` threads of `kernel` that are resident on all SMs at once
// (occupancy API, cached per kernel): the grid of a persistent grid-stride
// kernel, so no CTA waits for a second wave.
int resident_grid(const void* kernel, int threads, int num_sms);

// Exclusive scan of nseg segments.  Segment s reads in[s*in_stride + i] for
// i < len(s) and writes out[s*out_stride + i]; len(s) = d_len[s] when d_len is
// non-null, else const_len.  With write_end, out[s*out_stride + len(s)] gets
// the segment total; seg_total (if non-null) gets it too.  max_len bounds
// every len(s).  scratch needs scan_scratch_elems(nseg, max_len) int64s,
// zeroed once before first use (the scan leaves its tickets at zero again).
int64_t scan_scratch_elems(int64_t nseg, int64_t max_len);

template <typename InT, typename OutT>
cudaError_t seg_scan(const InT* in, int64_t in_stride, OutT* out, int64_t out_stride,
                     const int32_t* d_len, int64_t const_len, int32_t nseg, int64_t max_len,
                     bool write_end, int32_t* seg_total, int64_t* scratch,
                     const int32_t* status, cudaStream_t st);

// Single-pass exclusive scan of n int32 values (decoupled look-back): out[i]
// = sum of in[i'] for i' < i; with write_end out[n] = the total; total_out
// (if non-null) gets it too.  in and out 16-byte aligned
// (flat_scan_supported).  scratch needs flat_scan_scratch_elems(n) uint64s,
// zero before first use (the scan leaves it zero again).  Scans sharing a
// scratch must be ordered on one stream.
int64_t flat_scan_scratch_elems(int64_t max_n);
bool flat_scan_supported(const int32_t* in, const int32_t* out);
cudaError_t flat_scan(const int32_t* in, int32_t* out, int64_t n, bool write_end,
                      int32_t* total_out, uint64_t* scratch, int32_t* status, cudaStream_t st);

// Exclusive scan of n int32 cell counts into out (n + 1 entries, the total
// last): single pass where flat_scratch is given and the arrays allow it,
// else the three-phase seg_scan with scan_scratch.
inline cudaError_t cells_scan(const int32_t* in, int32_t* out, int64_t n, uint64_t* flat_scratch,
                              int64_t* scan_scratch, int32_t* status, cudaStream_t st) {
  if (flat_scratch && flat_scan_supported(in, out))
    return flat_scan(in, out, n, true, nullptr, flat_scratch, status, st);
  return seg_scan<int32_t, int32_t>(in, 0, out, 0, nullptr, n, 1, n, true, nullptr, scan_scratch,
                                    status, st);
}

// Exclusive scan down each column of a row-major [rows x cols] matrix:
// out[r*cols + c] = sum of in[r'*cols + c] over r' < r (coalesced along
// rows).  total_out[c] (if non-null) = column total + add_in[c] (add_in may be
// null).  scratch needs col_scan_scratch_elems(rows, cols) int64s.
int64_t col_scan_scratch_elems(int64_t rows, int32_t cols);
cudaError_t col_scan(const int32_t* in, int32_t* out, int64_t rows, int32_t cols,
                     const int32_t* add_in, int32_t* total_out, int64_t* scratch,
                     const int32_t* status, cudaStream_t st);

// ---- blocks.cu -------------------------------------------------------------
struct BlockTables {
  int32_t* start_node = nullptr;   // first node of each block start
  int32_t* start_block = nullptr;  // block index of each start
  int64_t n_starts = 0;
  int64_t n_blocks = 0;            // incl. continuation blocks of split objects
  int32_t* tile_first = nullptr;   // T+1
  int32_t* chunk_tile = nullptr;   // C+1
  int32_t* tile_adj_block = nullptr;
  int32_t* tile_feat_block = nullptr;
  int32_t* fblock_first_tile = nullptr;  // n_feat_blocks+1: first tile of each feature block
  int32_t* tile_adj_start = nullptr;     // T: block start (run) index of each tile
  int32_t* run_first_tile = nullptr;     // n_starts+1: first tile of each block run
  int64_t* blk_e0 = nullptr;             // n_blocks: first edge held by each physical block
  int64_t* blk_e1 = nullptr;             // n_blocks: one past its last edge
  int64_t T = 0;
  int64_t n_feat_blocks = 0;
  int64_t rows_per_feat_block = 0;
};

// Builds the block tables on the device; allocates the arrays in *bt.
cudaError_t build_block_tables(const void* d_offsets, int offsets_bits, int64_t N, int64_t E,
                               int64_t adj_block_bytes, int64_t rows_per_feat_block,
                               BlockTables* bt, cudaStream_t st, char* err, size_t errlen);
void free_block_tables(BlockTables* bt);

// ---- sample.cu -------------------------------------------------------------
struct HopArgs {
  // graph
  const void* offsets;
  int offsets_bits;
  const int32_t* indices;
  int32_t N;
  // tiles
  const int32_t* tile_first;
  const int32_t* chunk_tile;
  int32_t T;
  // hyperbatch shape
  int32_t H;
  int64_t capK;      // node capacity per minibatch
  int64_t cap_prev;  // frontier capacity per minibatch at this hop
  int64_t ecap;      // edge capacity per minibatch at this hop
  int32_t k;         // fanout
  int32_t hop;       // 1-based
  const uint64_t* key;  // device: {seed, first minibatch id} (launch_set_key)
  int32_t* status;
  // fanouts above kWideMax: per-warp hash sets of chosen positions, 2^hset_log2
  // int32 entries each, for the hset_grid CTAs of the sampler
  int32_t* hset = nullptr;
  int32_t hset_log2 = 0;
  int32_t hset_grid = 0;
  // the sampled bucket holds 4-byte entries (edge index << 12 | tile-local
  // id): the default frontier with ecap <= kPackedEdgeMax; the sampler then
  // records rank << 12 | tile-local id per edge (no rank array)
  bool sb_packed = false;
  // per frontier entry (bucket order): its node's first edge and degree, two
  // int64 each, written by the count kernel and read by the fill
  int64_t* fbd = nullptr;
};

constexpr int64_t kPackedEdgeMax = (int64_t)1 << 20;

// The hash sets the sampler needs for a fanout k > kWideMax: 2^log2 >= 2k
// entries per warp and the CTAs of its grid (capped so the tables stay within
// 1 GiB); returns the int32 entries to allocate (0 when k <= kWideMax).
int64_t huge_fanout_tables(int32_t k, int num_sms, int32_t* log2, int32_t* grid);

// Writes the sampling key {seed, first minibatch id} to device memory ahead
// of a hyperbatch (one 1-thread kernel: the arguments travel with the launch).
cudaError_t launch_set_key(uint64_t* key, uint64_t seed, uint64_t first_gid, cudaStream_t st);

cudaError_t launch_bucket_targets(int32_t* nodes, int64_t capK, int32_t H, int32_t B, int32_t N,
                                  const int32_t* tile_first, const int32_t* chunk_tile, int32_t T,
                                  int32_t* fcnt, int32_t* fcell_off, int32_t* tmp_id,
                                  int32_t* tmp_pos, int32_t* fb_id, int32_t* fb_pos,
                                  int64_t* scan_scratch, uint64_t* flat_scratch, int32_t* status,
                                  int num_sms, cudaStream_t st);

cudaError_t launch_sample_count(const HopArgs& a, const int32_t* fb_id, const int32_t* fb_pos,
                                const int32_t* fcell_off, int32_t* cnt, int num_sms,
                                cudaStream_t st);

// Which frontier cells to sample and, for streamed topology, where their
// edge lists are (gbuf == nullptr: the edges are read from HopArgs::indices).
struct FillRange {
  int64_t cell_lo = 0, cell_hi = 0;
  const int32_t* tile_adj_block = nullptr;
  const int32_t* blk_slot = nullptr;
  const int64_t* blk_e0 = nullptr;
  const int32_t* gbuf = nullptr;
  int64_t epb = 0, bb = 0;
  // gbuf is a topology cache: a block without a slot is read in place from
  // HopArgs::indices (otherwise every needed block must have a slot)
  bool in_place_fallback = false;
};

// Samples the frontier entries of cells [r.cell_lo, r.cell_hi) and records,
// per sampled edge, its neighbour id (nbr), its (tile, minibatch) cell (scell)
// and its rank within that cell (srank), counting the cells in scnt.  With
// HopArgs::sb_packed, nbr holds rank << 12 | tile-local id and srank is not
// written.
cudaError_t launch_sample_fill(const HopArgs& a, const int32_t* fb_id, const int32_t* fb_pos,
                               const int32_t* fcell_off, const int64_t* indptr, int32_t* nbr,
                               int32_t* scnt, int32_t* scell, int32_t* srank,
                               const FillRange& r, int num_sms, cudaStream_t st);

// ---- dedup.cu --------------------------------------------------------------
// Cells with more than this many entries (frontier + sampled) are resolved
// on bitmaps, one warp each; the rest entry-parallel.  The big-cell list
// therefore holds at most (entries) / (kDedupSmallMax + 1) cells.
constexpr int kDedupSmallMax = 32;
// With the default frontier, cells of at most this many entries are resolved
// by one thread each; larger cells with samples are queued (q_dense), so the
// queue holds at most (entries) / (kDedupLaneMax + 1) cells.
constexpr int kDedupLaneMax = 8;
// The lane kernel's unit of dynamically scheduled work: 256 consecutive cells.
constexpr int kDedupChunkCells = 256;

struct DedupBufs {
  const int32_t* nbr;       // H x ecap sampled ids (packed: rank << 12 | tile-local id)
  const int32_t* ecnt;      // H edge counts
  const int32_t* scell;     // H x ecap: cell of each sampled id
  const int32_t* srank;     // H x ecap: its rank within the cell (not packed)
  const int32_t* scnt;      // T*H per-cell counts of sampled ids
  int32_t* soff;            // T*H+1
  int2* sb;                 // bucketed (sampled id, edge index in the minibatch), or packed
                            // 4-byte entries edge index << 12 | tile-local id (sb_packed)
  int2* tmp;                // per cell: next-frontier entries with local ranks
  int32_t* big_list;        // cells with more than kDedupSmallMax entries
  int32_t* big_n;           // their count
  // default frontier: the queue of cells with samples and more than
  // kDedupLaneMax entries: per chunk of kDedupChunkCells cells a run in
  // q_cells (T*H), the runs' counts and offsets (q_chunks_cap,
  // q_chunks_cap + 1), the queue in cell order (q_dense), and the lane
  // kernel's chunk counter (q_next, zero between launches)
  int32_t* q_cells;
  int32_t* q_cnt;
  int32_t* q_off;
  int32_t* q_dense;
  int32_t* q_next;
  int32_t q_chunks_cap;
  const int32_t* fb_id;     // current frontier bucket
  const int32_t* fb_pos;
  const int32_t* fcell_off;
  int32_t* newcnt;          // T*H: new ids per cell
  int32_t* newbase;         // T*H: per-minibatch exclusive scan of newcnt over tiles
  int32_t* nfcnt;           // T*H
  int32_t* nfcell_off;      // T*H+1
  int32_t* nfb_id;          // next frontier bucket
  int32_t* nfb_pos;
  const int32_t* nsz_prev;  // H frontier sizes
  int32_t* nsz_next;        // H: next frontier sizes
  int32_t* srcsz;           // H: |src_h| = |dst_h| + new ids
  int32_t* noutbase;        // T*H (frontier_sampled): per-minibatch scan of nfcnt over tiles
  bool frontier_sampled;    // next frontier = distinct sampled ids (Algorithm 1's N_out)
  int32_t* nodes;           // H x capK
  int32_t* col;             // H x ecap
  const int32_t* tile_adj_block;
  uint8_t* adj_flags;       // per topology block: touched at this hop
  int64_t* scan_scratch;
  uint64_t* flat_scratch = nullptr;  // flat_scan_scratch_elems(T*H), or null
  // If side is set, the new-id scan (into newbase, with side_scratch) and the
  // col fix-up (which needs only newbase, col and scell) run on it, forked
  // from st through the event fork; st waits for the scan through the event
  // ready, and the caller joins side back before anything rewrites scell,
  // newbase or the hop's col.
  cudaStream_t side = nullptr;
  cudaEvent_t fork = nullptr, ready = nullptr;
  int64_t* side_scratch = nullptr;  // col_scan_scratch_elems(T, H) int64
};

// One hop's dedup up to the next-frontier offsets (nfcell_off, nsz_next) and
// the new-id offsets (newbase): scatter, cells, big cells, scans, col fix-up.
cudaError_t launch_dedup(const HopArgs& a, const DedupBufs& d, int num_sms, cudaStream_t st);
// Then the compaction: the next frontier bucket (nfb_id / nfb_pos) and the
// new nodes' ids in the node lists.
cudaError_t launch_dedup_compact(const HopArgs& a, const DedupBufs& d, int num_sms,
                                 cudaStream_t st);

// ---- dedup_cells.cu --------------------------------------------------------
// The default frontier's resolution of one hop's cells (launch_dedup calls
// it in place of the sampled frontier's cell kernels): newcnt, nfcnt, col
// with local new-id ranks, the next frontier cells in tmp, the touched-block
// flags; it builds and uses the queue in q_cells / q_cnt / q_off / q_dense.
cudaError_t launch_dedup_cells(const HopArgs& a, const DedupBufs& d, int num_sms,
                               cudaStream_t st);

// ---- gather.cu -------------------------------------------------------------
cudaError_t launch_gather(const void* feats, int64_t row_bytes, const int32_t* fb_id,
                          const int32_t* fb_pos, const int32_t* total, void* out,
                          const int32_t* status, int num_sms, cudaStream_t st);

// Gathers the rows of a batch of feature blocks held in HBM copies: the
// batch's blocks are touched[0 .. nb) (ascending), block touched[p] starts at
// device address src[p]; its bucket entries are those of cells
// [cell_lo, cell_hi) of cell_off.  Rows must be a multiple of 16 bytes.
cudaError_t launch_gather_staged(const unsigned long long* src, int64_t row_bytes, int64_t rpb,
                                 const int32_t* touched, int32_t nb, const int32_t* fb_id,
                                 const int32_t* fb_pos, const int32_t* cell_off, int64_t cell_lo,
                                 int64_t cell_hi, void* out, const int32_t* status, int num_sms,
                                 cudaStream_t st);

// Gathers every row of the final bucket from its feature block's address:
// row v at (const uint4*)addr[v / rpb] + (v % rpb) * row_bytes / 16 (an HBM
// cache slot or mapped pinned host memory).  Rows must be a multiple of 16
// bytes.
cudaError_t launch_gather_table(const unsigned long long* addr, int64_t row_bytes, int64_t rpb,
                                const int32_t* fb_id, const int32_t* fb_pos, const int32_t* total,
                                void* out, const int32_t* status, int num_sms, cudaStream_t st);

// Row mode, de-duplicated (see gather.cu): per tile t, the bitmap of requested
// ids (kTileWords words at bitmap + t * kTileWords), the exclusive prefix of
// set bits per word (wpref) and their count (dcnt[t]).
cudaError_t launch_tile_bitmaps(const int32_t* fb_id, const int32_t* cell_off,
                                const int32_t* tile_first, int32_t T, int32_t H, uint32_t* bitmap,
                                uint16_t* wpref, int32_t* dcnt, const int32_t* status,
                                cudaStream_t st);
// Copies the distinct requested rows of tiles [t_lo, t_hi) (doff = exclusive
// scan of dcnt, T + 1 entries) of blocks outside the feature cache
// [cache_lo, cache_hi) from their block's address to staging, counting them
// in *host_rows; at most max_blocks CTAs.
cudaError_t launch_load_distinct_rows(const unsigned long long* addr, int64_t row_bytes,
                                      int64_t rpb, const uint32_t* bitmap, const uint16_t* wpref,
                                      const int32_t* doff, int32_t t_lo, int32_t t_hi,
                                      const int32_t* tile_first, void* staging,
                                      unsigned long long cache_lo, unsigned long long cache_hi,
                                      unsigned long long* host_rows, const int32_t* status,
                                      int max_blocks, int num_sms, cudaStream_t st);
// Gathers the entries [*lo, *hi) of the final bucket from the staging row of
// their id, or in place from the feature cache when its block's address (addr,
// one per feature block of rpb rows) lies in [cache_lo, cache_hi).
cudaError_t launch_gather_staged_rows(const void* staging, int64_t row_bytes, const int32_t* fb_id,
                                      const int32_t* fb_pos, const int32_t* lo, const int32_t* hi,
                                      const int32_t* tile_first, const int32_t* chunk_tile,
                                      int32_t T, const uint32_t* bitmap, const uint16_t* wpref,
                                      const int32_t* doff, const unsigned long long* addr,
                                      int64_t rpb, unsigned long long cache_lo,
                                      unsigned long long cache_hi, void* out,
                                      const int32_t* status, int num_sms, cudaStream_t st);

// Copies feature blocks blk[0 .. njobs) (block_bytes each, the last block of
// the matrix possibly shorter) from host_dev, the device view of pinned host
// memory holding host_bytes bytes, to device addresses dst[0 .. njobs).
// block_bytes, host_bytes and every address must be multiples of 16.
cudaError_t launch_load_feat_blocks(const void* host_dev, int64_t host_bytes, const int32_t* blk,
                                    const unsigned long long* dst, int32_t njobs,
                                    int64_t block_bytes, int num_sms, cudaStream_t st);

// Marks flags[map[t]] for every tile t whose cells (t, 0..H-1) in cell_off
// hold an entry, then counts set flags into *count (int64).
cudaError_t launch_mark_count(const int32_t* cell_off, int32_t T, int32_t H, const int32_t* map,
                              uint8_t* flags, int64_t n_flags, int64_t* count,
                              const int32_t* status, cudaStream_t st);

// Topology cache bookkeeping for one hop's frontier bucket: acc[run] +=
// requests of the block run's tiles; cached += requests on tiles whose
// topology block has a cache slot.  Both accumulate since load.
cudaError_t launch_count_cache_requests(const int32_t* cell_off, int32_t T, int32_t H,
                                        const int32_t* tile_adj_start,
                                        const int32_t* tile_adj_block, const int32_t* blk_slot,
                                        unsigned long long* acc, unsigned long long* cached,
                                        const int32_t* status, cudaStream_t st);

// counts[tile_map[t]] += requests (bucket entries) of tile t, for every tile:
// per feature block (tile_feat_block) or per topology block run
// (tile_adj_start).  zero_first clears the n counts first.
cudaError_t launch_count_requests(const int32_t* cell_off, int32_t T, int32_t H,
                                  const int32_t* tile_map, int32_t* counts, int64_t n,
                                  bool zero_first, const int32_t* status, cudaStream_t st);

// Copies physical blocks jobs[i].x (edges e0..e1 of host_indices, a device
// view of pinned host memory) into graph-buffer slots jobs[i].y.
cudaError_t launch_load_blocks(const int32_t* host_indices, const int64_t* e0, const int64_t* e1,
                               const int2* jobs, int32_t njobs, int32_t* gbuf, int64_t epb,
                               int num_sms, cudaStream_t st);

// need[r] = 1 for every block run r whose tiles hold a frontier entry
// (need is cleared first).
cudaError_t launch_mark_runs(const int32_t* cell_off, int32_t T, int32_t H,
                             const int32_t* tile_adj_start, uint8_t* need, int64_t n_runs,
                             const int32_t* status, cudaStream_t st);

cudaError_t launch_distinct_rows(const int32_t* fb_id, const int32_t* cell_off,
                                 const int32_t* tile_first, int32_t T, int32_t H,
                                 unsigned long long* count, cudaStream_t st);

// Makes `device` current for the lifetime of the guard and then restores the
// device that was current when it was made, so that an entry point never
// leaves the calling thread on another GPU.
class DeviceGuard {
 public:
  explicit DeviceGuard(int device) {
    if (cudaGetDevice(&prev_) != cudaSuccess) {
      cudaGetLastError();
      prev_ = -1;
    }
    ok_ = prev_ == device || cudaSetDevice(device) == cudaSuccess;
    if (!ok_) cudaGetLastError();
    switched_ = ok_ && prev_ >= 0 && prev_ != device;
  }
  ~DeviceGuard() {
    if (switched_) cudaSetDevice(prev_);
  }
  DeviceGuard(const DeviceGuard&) = delete;
  DeviceGuard& operator=(const DeviceGuard&) = delete;
  bool ok() const { return ok_; }

 private:
  int prev_ = -1;
  bool ok_ = false;
  bool switched_ = false;
};

// ---- api.cu: read-only view of a loaded graph for other translation units --
struct GraphView {
  int device;
  int num_sms;
  const void* offsets;
  int offsets_bits;
  int64_t N;
};

}  // namespace agnes

struct agnes_ctx;
void ctx_graph_view(const agnes_ctx* ctx, agnes::GraphView* out);
void ctx_set_error(agnes_ctx* ctx, const char* fmt, ...);
// A device buffer owned by ctx of at least `bytes` (grown on demand, freed by
// agnes_free); its contents do not outlive the call that asked for it.
cudaError_t ctx_scratch(agnes_ctx* ctx, size_t bytes, void** out);
// The same for pinned host memory (staging for small host <-> device copies).
cudaError_t ctx_pinned(agnes_ctx* ctx, size_t bytes, void** out);
