// prepare.cu -- agnes_prepare_hyperbatch: one hyperbatch (Algorithm 1,
// Sec. 3.5) on the caller's stream:
//   bucket the targets by (tile, minibatch)                   [sample.cu]
//   for each hop: count min(deg, k) per frontier entry, scan to indptr,
//                 sample in bucket order                      [sample.cu, scan.cu]
//                 bucket the samples, dedup + relabel, carry the bucket
//                                                             [dedup.cu]
//   gather the final bucket's rows block by block             [gather_hbm.cu]
//   count the blocks touched (the paper's block-wise I/Os)   [gather.cu]
// Everything is sized for the worst case up front (per-minibatch capacities
// cap_h = min(N, B * prod(1 + k))), so no kernel's launch waits on a count
// from the device and the host synchronises only when a view is fetched.
// With the graph resident the sequence is captured once per hyperbatch shape
// and replayed as one CUDA graph launch.
#include <string.h>

#include <utility>
#include <vector>

#include "ctx.h"

using namespace agnes;

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

void free_workspace(Workspace* w) {
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
  cudaFree(w->q_cells);
  cudaFree(w->hset);
  cudaFree(w->q_cnt);
  cudaFree(w->q_off);
  cudaFree(w->q_next);
  cudaFree(w->q_dense);
  cudaFree(w->big_n);
  cudaFree(w->tmp_id);
  cudaFree(w->tmp_pos);
  cudaFree(w->cnt);
  cudaFree(w->fbd);
  cudaFree(w->flat_scratch);
  cudaFree(w->feats_out);
  cudaFree(w->adj_flags);
  cudaFree(w->feat_flags);
  cudaFree(w->stats);
  cudaFree(w->scan_scratch);
  cudaFree(w->side_scratch);
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
  w.q_chunks_cap = (int32_t)((cells + kDedupChunkCells - 1) / kDedupChunkCells);
  WA(w.q_cells, cells);
  WA(w.q_cnt, w.q_chunks_cap);
  WA(w.q_off, w.q_chunks_cap + 1);
  WA(w.q_next, 1);
  WA(w.q_dense, (rows + edges) / (kDedupLaneMax + 1) + 1);
  w.hset_elems = 0;
  for (int h = 0; h < K; ++h) {
    int32_t l2 = 0, g = 0;
    const int64_t e = huge_fanout_tables(fan[h], ctx->num_sms, &l2, &g);
    if (e > w.hset_elems) w.hset_elems = e;
  }
  if (w.hset_elems > 0) WA(w.hset, w.hset_elems);
  WA(w.tmp_id, (int64_t)H * B);
  WA(w.tmp_pos, (int64_t)H * B);
  WA(w.cnt, (int64_t)H * w.cap_prev_max);
  WA(w.fbd, 2 * (int64_t)H * w.cap_prev_max);
  w.flat_elems = flat_scan_scratch_elems(cells);
  WA(w.flat_scratch, w.flat_elems);
  {
    uint8_t* f = nullptr;
    WA(f, rows * ctx->row_bytes);
    w.feats_out = f;
  }
  WA(w.adj_flags, (int64_t)K * nb);
  WA(w.feat_flags, nfb);
  WA(w.stats, K + 1);
  WA(w.scan_scratch, scratch);
  WA(w.side_scratch, s4);
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
      cudaMemset(w.side_scratch, 0, sizeof(int64_t) * s4) != cudaSuccess ||
      cudaMemset(w.fcnt, 0, sizeof(int32_t) * cells) != cudaSuccess ||
      cudaMemset(w.scnt, 0, sizeof(int32_t) * cells) != cudaSuccess ||
      cudaMemset(w.q_next, 0, sizeof(int32_t)) != cudaSuccess ||
      cudaMemset(w.flat_scratch, 0, sizeof(uint64_t) * w.flat_elems) != cudaSuccess) {
    free_workspace(&w);
    set_err(ctx, "cudaMemset failed");
    return AGNES_ECUDA;
  }
  w.valid = true;
  return AGNES_OK;
}

void swap_hyperbatch_state(agnes_ctx* ctx, agnes_ctx::Spare& o) {
  std::swap(ctx->ws, o.ws);
  std::swap(ctx->lg, o.lg);
  std::swap(ctx->ws_gen, o.ws_gen);
  std::swap(ctx->done, o.done);
  std::swap(ctx->aux_fork, o.aux_fork);
  std::swap(ctx->aux_join, o.aux_join);
  std::swap(ctx->aux_ready, o.aux_ready);
  std::swap(ctx->aux, o.aux);
  std::swap(ctx->pipe_st, o.pipe_st);
  std::swap(ctx->cur, o.cur);
  std::swap(ctx->prepared, o.prepared);
  std::swap(ctx->synced, o.synced);
}

void rotate_hyperbatch_state(agnes_ctx* ctx) {
  swap_hyperbatch_state(ctx, ctx->spares[0]);
  for (int i = 0; i + 2 < ctx->pipe_depth; ++i) std::swap(ctx->spares[i], ctx->spares[i + 1]);
}

static agnes_status make_one_spare(agnes_ctx* ctx, agnes_ctx::Spare& o) {
  if (o.done) return AGNES_OK;
  const unsigned f = cudaEventDisableTiming;
  if (cudaEventCreateWithFlags(&o.done, f) != cudaSuccess ||
      cudaEventCreateWithFlags(&o.aux_fork, f) != cudaSuccess ||
      cudaEventCreateWithFlags(&o.aux_join, f) != cudaSuccess ||
      cudaEventCreateWithFlags(&o.aux_ready, f) != cudaSuccess ||
      cudaStreamCreateWithFlags(&o.aux, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&o.pipe_st, cudaStreamNonBlocking) != cudaSuccess) {
    cudaGetLastError();
    set_err(ctx, "creating a further hyperbatch's events or streams failed");
    return AGNES_ECUDA;
  }
  o.lg.mode = ctx->lg.mode;
  return AGNES_OK;
}

agnes_status make_spare_state(agnes_ctx* ctx, int32_t depth) {
  for (int i = 0; i + 1 < depth; ++i) {
    const agnes_status rc = make_one_spare(ctx, ctx->spares[i]);
    if (rc != AGNES_OK) return rc;
  }
  const unsigned f = cudaEventDisableTiming;
  if ((!ctx->pipe_st && cudaStreamCreateWithFlags(&ctx->pipe_st, cudaStreamNonBlocking) !=
                            cudaSuccess) ||
      (!ctx->pipe_in && cudaEventCreateWithFlags(&ctx->pipe_in, f) != cudaSuccess)) {
    cudaGetLastError();
    set_err(ctx, "creating the pipeline's stream or event failed");
    return AGNES_ECUDA;
  }
  return AGNES_OK;
}

void free_spare_state(agnes_ctx* ctx) {
  for (agnes_ctx::Spare& o : ctx->spares) {
    drop_launch_graph(&o.lg);
    if (o.lg.cap) cudaStreamDestroy(o.lg.cap);
    o.lg.cap = nullptr;
    free_workspace(&o.ws);
    if (o.done) cudaEventDestroy(o.done);
    if (o.aux_fork) cudaEventDestroy(o.aux_fork);
    if (o.aux_join) cudaEventDestroy(o.aux_join);
    if (o.aux_ready) cudaEventDestroy(o.aux_ready);
    if (o.aux) cudaStreamDestroy(o.aux);
    if (o.pipe_st) cudaStreamDestroy(o.pipe_st);
    const int32_t mode = o.lg.mode;
    o = agnes_ctx::Spare();
    o.lg.mode = mode;
  }
}

void drop_launch_graph(agnes_ctx::LaunchGraph* g) {
  if (g->exec) cudaGraphExecDestroy(g->exec);
  if (g->graph) cudaGraphDestroy(g->graph);
  g->exec = nullptr;
  g->graph = nullptr;
  g->n_marks = 0;
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
  // a phase boundary; with AGNES_PROFILE_GATHER only the gather's two count
  auto mark = [&](bool gather_edge = false) {
    if (ctx->profiling == AGNES_PROFILE_PHASES ||
        (ctx->profiling == AGNES_PROFILE_GATHER && gather_edge))
      cudaEventRecordWithFlags(ctx->ev[ring][ph++], st, mark_flags);
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
                                w.fb_id[0], w.fb_pos[0], w.scan_scratch, w.flat_scratch, w.status,
                                nsm, st));
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
    a.hset = w.hset;
    a.fbd = w.fbd;
    huge_fanout_tables(fanouts[h], nsm, &a.hset_log2, &a.hset_grid);
    const bool frontier_sampled = ctx->frontier_mode == AGNES_FRONTIER_SAMPLED && h + 1 < K;
    a.sb_packed = !frontier_sampled && a.ecap <= kPackedEdgeMax;
    int32_t* nsz_prev = w.nsz + (int64_t)h * H;
    int32_t* ecnt = w.ecnt + (int64_t)h * H;
    CK(ctx, launch_sample_count(a, w.fb_id[cur], w.fb_pos[cur], w.fcell_off[cur], w.cnt, nsm, st));
    CK(ctx, (seg_scan<int32_t, int64_t>(w.cnt, cap[h], w.indptr[h], cap[h] + 1, nsz_prev, 0, H,
                                         cap[h], true, ecnt, w.scan_scratch, w.status, st)));
    mark();
    CK(ctx, cudaMemsetAsync(w.scnt, 0, sizeof(int32_t) * cells, st));
    // the previous hop's col fix-up still reads scell and newbase
    if (h > 0) {
      CK(ctx, cudaEventRecord(ctx->aux_join, ctx->aux));
      CK(ctx, cudaStreamWaitEvent(st, ctx->aux_join, 0));
    }
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
    d.q_cells = w.q_cells;
    d.q_cnt = w.q_cnt;
    d.q_off = w.q_off;
    d.q_dense = w.q_dense;
    d.q_next = w.q_next;
    d.q_chunks_cap = w.q_chunks_cap;

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
    d.frontier_sampled = frontier_sampled;
    d.nodes = w.nodes;
    d.col = w.col[h];
    d.tile_adj_block = ctx->bt.tile_adj_block;
    d.adj_flags = w.adj_flags + (int64_t)h * ctx->bt.n_blocks;
    d.scan_scratch = w.scan_scratch;
    d.flat_scratch = w.flat_scratch;
    d.side = ctx->aux;
    d.fork = ctx->aux_fork;
    d.ready = ctx->aux_ready;
    d.side_scratch = w.side_scratch;
    CK(ctx, launch_dedup(a, d, nsm, st));
    if (h + 1 == K) {
      // blocks touched by the hyperbatch (the statistics), on the side stream
      // beside the last compaction: feature blocks from the final bucket's
      // offsets, topology blocks from the flags the dedup of each hop set
      CK(ctx, cudaEventRecord(ctx->aux_fork, st));
      CK(ctx, cudaStreamWaitEvent(ctx->aux, ctx->aux_fork, 0));
      CK(ctx, launch_mark_count(w.fcell_off[1 - cur], T, H, ctx->bt.tile_feat_block, w.feat_flags,
                                ctx->bt.n_feat_blocks, w.stats + K, w.status, ctx->aux));
      for (int hh = 0; hh < K; ++hh)
        CK(ctx, launch_mark_count(nullptr, T, H, nullptr,
                                  w.adj_flags + (int64_t)hh * ctx->bt.n_blocks, ctx->bt.n_blocks,
                                  w.stats + hh, w.status, ctx->aux));
    }
    CK(ctx, launch_dedup_compact(a, d, nsm, st));
    cur = 1 - cur;
  }
  mark(true);
  if (ctx->features_on_host) {
    rc = gather_streamed(ctx, cur, st);
    if (rc != AGNES_OK) return rc;
  } else {
    CK(ctx, launch_gather(ctx->features, ctx->row_bytes, w.fb_id[cur], w.fb_pos[cur],
                          w.fcell_off[cur] + cells, w.feats_out, w.status, nsm, st));
  }
  mark(true);
  // the last hop's col fix-up and the statistics ran beside its compaction
  CK(ctx, cudaEventRecord(ctx->aux_join, ctx->aux));
  CK(ctx, cudaStreamWaitEvent(st, ctx->aux_join, 0));
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

// Turns every kernel-to-kernel link of the captured chain (an edge whose
// source has no other successor and whose destination no other predecessor;
// fork and join edges of the side stream stay as they are) into a
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
  std::vector<std::pair<cudaGraphNode_t, int>> outs, ins;  // edge counts per node
  auto bump = [](std::vector<std::pair<cudaGraphNode_t, int>>& v, cudaGraphNode_t nd) {
    for (auto& p : v)
      if (p.first == nd) return ++p.second;
    v.emplace_back(nd, 1);
    return 1;
  };
  auto count = [](const std::vector<std::pair<cudaGraphNode_t, int>>& v, cudaGraphNode_t nd) {
    for (const auto& p : v)
      if (p.first == nd) return p.second;
    return 0;
  };
  for (size_t i = 0; i < n; ++i) {
    bump(outs, from[i]);
    bump(ins, to[i]);
  }
  for (size_t i = 0; i < n; ++i) {
    if (count(outs, from[i]) != 1 || count(ins, to[i]) != 1) continue;
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

extern "C" {

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
  if ((int64_t)H * ctx->bt.T >= lim) {  // cell indices are 31-bit in the kernels
    set_err(ctx, "H x tiles (%lld) exceeds 2^31", (long long)(H * ctx->bt.T));
    return AGNES_ERANGE;
  }
  DeviceGuard dg(ctx->device);
  if (!dg.ok()) {
    set_err(ctx, "cudaSetDevice(%d) failed", ctx->device);
    return AGNES_ECUDA;
  }
  cudaStream_t st = (cudaStream_t)cuda_stream;
  const bool capturing = stream_capturing(st);
  const bool resident = !ctx->features_on_host && !ctx->topo.on;
  const bool pipelined = ctx->pipe_depth > 1 && resident && !capturing;
  if (pipelined) {
    // the least recently used set of per-hyperbatch state: its internal
    // stream starts once the caller's stream reaches this call, and is
    // already ordered after the set's previous hyperbatch
    rotate_hyperbatch_state(ctx);
    CK(ctx, cudaEventRecord(ctx->pipe_in, st));
    CK(ctx, cudaStreamWaitEvent(ctx->pipe_st, ctx->pipe_in, 0));
    st = ctx->pipe_st;
  }
  agnes_status rc = ensure_workspace(ctx, H, B, fanouts, K, cap);
  if (rc != AGNES_OK) return rc;
  Workspace& w = ctx->ws;
  ctx->prepared = false;
  ctx->synced = false;
  if (ctx->profiling && !ctx->ev_created) {
    for (int r = 0; r < kEventRing; ++r)
      for (int i = 0; i <= kMaxPhases; ++i) CK(ctx, cudaEventCreate(&ctx->ev[r][i]));
    ctx->ev_created = true;
  }
  const int ring = (int)(ctx->n_prepared % kEventRing);
  ctx->n_phases[ring] = 0;
  // a prepare on another stream than the last one on these buffers still runs
  // after it (a caller's own capture orders its replays itself)
  if (ctx->n_prepared > 0 && !capturing) CK(ctx, cudaStreamWaitEvent(st, ctx->done, 0));
  if (!capturing) {
    rc = update_topology_cache(ctx, st);
    if (rc != AGNES_OK) return rc;
  }
  CK(ctx, cudaMemcpy2DAsync(w.nodes, sizeof(int32_t) * w.capK, targets, sizeof(int32_t) * B,
                            sizeof(int32_t) * B, H, cudaMemcpyDefault, st));
  CK(ctx, launch_set_key(w.key, seed, first_minibatch_id, st));
  int n_marks = 0;
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

}  // extern "C"
