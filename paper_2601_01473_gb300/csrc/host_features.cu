// host_features.cu -- the gather with features in pinned host memory
// (features_on_host): block I/O through a ring of HBM staging slots, row I/O
// in place over the host link, and the count-based feature cache (Sec. 3.3,
// Sec. 3.4 (2) and (4)).
#include <string.h>

#include <algorithm>
#include <vector>

#include "ctx.h"

using namespace agnes;

// Staging ring (block mode), feature cache, copy stream and host tables for
// host-resident features.
agnes_status setup_streaming(agnes_ctx* ctx, const agnes_graph_desc* d, cudaStream_t st) {
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
  for (int i = 0; i < kRowChunks; ++i)
    CK(ctx, cudaEventCreateWithFlags(&ctx->rows_loaded[i], cudaEventDisableTiming));
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
// staging slots.  Batch by batch, a loader kernel on the copy stream reads
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
  // The rows are loaded on the copy stream in kRowChunks tile ranges, and each
  // range's gather (HBM-bound) runs on st once its rows are in, overlapping
  // the next range's load (bound by the host link).  The loads start when st
  // gets here: the bitmaps are built, and the previous hyperbatch's gathers
  // no longer read the staging rows.  The loader is held to four CTAs per SM,
  // enough rows in flight for the link, so the gathers find room beside it.
  CK(ctx, cudaEventRecord(ctx->gather_start, st));
  CK(ctx, cudaStreamWaitEvent(ctx->copy_stream, ctx->gather_start, 0));
  for (int c = 0; c < kRowChunks; ++c) {
    const int32_t t_lo = (int32_t)((int64_t)T * c / kRowChunks);
    const int32_t t_hi = (int32_t)((int64_t)T * (c + 1) / kRowChunks);
    if (t_hi <= t_lo) continue;
    CK(ctx, launch_load_distinct_rows(ctx->d_addr, rb, rpb, ctx->rm_bitmap, ctx->rm_wpref,
                                      ctx->rm_doff, t_lo, t_hi, ctx->bt.tile_first,
                                      ctx->rm_staging, 0, 0, ctx->d_host_rows, w.status,
                                      4 * ctx->num_sms, ctx->num_sms, ctx->copy_stream));
    CK(ctx, cudaEventRecord(ctx->rows_loaded[c], ctx->copy_stream));
    CK(ctx, cudaStreamWaitEvent(st, ctx->rows_loaded[c], 0));
    CK(ctx, launch_gather_staged_rows(ctx->rm_staging, rb, w.fb_id[cur], w.fb_pos[cur],
                                      w.fcell_off[cur] + (int64_t)t_lo * w.H,
                                      w.fcell_off[cur] + (int64_t)t_hi * w.H, ctx->bt.tile_first,
                                      ctx->bt.chunk_tile, T, ctx->rm_bitmap, ctx->rm_wpref,
                                      ctx->rm_doff, ctx->d_addr, rpb, 0, 0, w.feats_out,
                                      w.status, ctx->num_sms, st));
  }
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
agnes_status gather_streamed(agnes_ctx* ctx, int cur, cudaStream_t st) {
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
