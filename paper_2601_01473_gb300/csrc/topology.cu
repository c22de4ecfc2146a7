// topology.cu -- sampling with the neighbour lists in pinned host memory
// (topology_on_host): the HBM graph buffer with LRU + pinning and waves of
// block loads (Sec. 3.4 (1)), and the topology cache of in-place reads.
#include <string.h>

#include <algorithm>
#include <vector>

#include "ctx.h"

using namespace agnes;

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
agnes_status setup_topology_cache(agnes_ctx* ctx, const agnes_graph_desc* d,
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

// Graph buffer, tables and copy stream for topology in pinned host memory
// with block I/O.
agnes_status setup_topology(agnes_ctx* ctx, const agnes_graph_desc* d, cudaStream_t st) {
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

// Sampling with the topology in pinned host memory.  The block runs the
// frontier touches are read back; runs are taken in order (ascending and
// descending in turn, hop by hop) into waves that fit the graph buffer: each
// needed block is either resident (a hit: pinned and moved to the recent end
// of the LRU list) or copied into the least recently used unpinned slot on
// the topology's copy stream.  The slot table
// is uploaded, the wave's cells are sampled, and the wave's blocks unpin when
// the next wave starts (its copies wait for this wave's sampling to finish).
agnes_status fill_streamed(agnes_ctx* ctx, const HopArgs& a, int cur, int h,
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

// Before hyperbatches 2, 2 + R, 2 + 2R, ... (R = kTopoRepickEvery) with a
// topology cache: waits for the previous hyperbatch, reads back the request
// count of every block run since load, and re-picks the cached runs -- most
// requested first, whole runs, up to the cache's capacity.  Runs that stay
// keep their slots; the blocks of newly admitted runs are copied into free
// slots (loader kernel over the host link) and the slot table is uploaded,
// all on st ahead of the hyperbatch.  Re-picking only every R hyperbatches
// keeps the wait (an idle GPU while the host plans) and the churn rare.
agnes_status update_topology_cache(agnes_ctx* ctx, cudaStream_t st) {
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
