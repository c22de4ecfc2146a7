// api.cu -- the C ABI of libagnes.so (declared in include/agnes.h): graph
// load and release, the views of a prepared hyperbatch, its statistics and
// counters, and the per-ctx settings.  agnes_prepare_hyperbatch is in
// prepare.cu; the host-resident modes are in host_features.cu and
// topology.cu (ctx.h has the context they share).
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <new>

#include "ctx.h"

using namespace agnes;

static thread_local char g_err[512];

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

static agnes_status wait_prepared(agnes_ctx* ctx) {
  if (!ctx) return AGNES_EINVAL;
  if (!ctx->prepared) {
    set_err(ctx, "no hyperbatch has been prepared");
    return AGNES_ESTATE;
  }
  if (!ctx->synced) {
    DeviceGuard dg(ctx->device);
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
    if (s & kErrWaitTimeout) {
      set_err(ctx, "a bounded wait between CTAs ran out (device status word 0x%x)", s);
      return AGNES_ETIMEOUT;
    }
    set_err(ctx, "device status word 0x%x", s);
    return AGNES_EKERNEL;
  }
  return AGNES_OK;
}

// ============================================================================
// Public API
// ============================================================================

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
  DeviceGuard dg(ctx->device);
  cudaDeviceSynchronize();
  drop_launch_graph(&ctx->lg);
  if (ctx->lg.cap) cudaStreamDestroy(ctx->lg.cap);
  free_workspace(&ctx->ws);
  free_spare_state(ctx);
  if (ctx->pipe_st) cudaStreamDestroy(ctx->pipe_st);
  if (ctx->pipe_in) cudaEventDestroy(ctx->pipe_in);
  free_block_tables(&ctx->bt);
  if (ctx->own_offsets) cudaFree(ctx->offsets);
  if (ctx->own_indices) cudaFree(ctx->indices);
  if (ctx->own_features) cudaFree(ctx->features);
  if (ctx->done) cudaEventDestroy(ctx->done);
  if (ctx->aux_fork) cudaEventDestroy(ctx->aux_fork);
  if (ctx->aux_join) cudaEventDestroy(ctx->aux_join);
  if (ctx->aux_ready) cudaEventDestroy(ctx->aux_ready);
  if (ctx->aux) cudaStreamDestroy(ctx->aux);
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
  for (int i = 0; i < kRowChunks; ++i)
    if (ctx->rows_loaded[i]) cudaEventDestroy(ctx->rows_loaded[i]);
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
  DeviceGuard dg(device);
  if (!dg.ok()) {
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
  if (rc == AGNES_OK && (cudaEventCreateWithFlags(&ctx->done, cudaEventDisableTiming) != cudaSuccess ||
                         cudaEventCreateWithFlags(&ctx->aux_fork, cudaEventDisableTiming) != cudaSuccess ||
                         cudaEventCreateWithFlags(&ctx->aux_join, cudaEventDisableTiming) != cudaSuccess ||
                         cudaEventCreateWithFlags(&ctx->aux_ready, cudaEventDisableTiming) != cudaSuccess ||
                         cudaStreamCreateWithFlags(&ctx->aux, cudaStreamNonBlocking) != cudaSuccess)) {
    cudaGetLastError();
    set_err(ctx, "creating events or the side stream failed");
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
  for (agnes_ctx::Spare& o : ctx->spares) o.lg.mode = mode;
  return AGNES_OK;
}

agnes_status agnes_set_pipeline_depth(agnes_ctx* ctx, int32_t depth) {
  if (!ctx) return AGNES_EINVAL;
  if (depth < 1 || depth > AGNES_MAX_PIPELINE_DEPTH) {
    set_err(ctx, "pipeline depth must be 1 .. %d", AGNES_MAX_PIPELINE_DEPTH);
    return AGNES_EINVAL;
  }
  if (depth > 1 && (ctx->features_on_host || ctx->topo.on)) {
    set_err(ctx, "a pipeline depth above 1 needs the graph resident in device memory");
    return AGNES_EINVAL;
  }
  if (depth == ctx->pipe_depth) return AGNES_OK;
  DeviceGuard dg(ctx->device);
  CK(ctx, cudaDeviceSynchronize());
  // the spare sets restart empty (the active set keeps the last hyperbatch)
  free_spare_state(ctx);
  if (depth > 1) {
    const agnes_status rc = make_spare_state(ctx, depth);
    if (rc != AGNES_OK) return rc;
  }
  ctx->pipe_depth = depth;
  return AGNES_OK;
}

agnes_status agnes_fetch_previous_hyperbatch(agnes_ctx* ctx, agnes_hyperbatch_view* out) {
  if (!ctx || !out) {
    set_err(ctx, "ctx and out must be non-NULL");
    return AGNES_EINVAL;
  }
  if (ctx->pipe_depth < 2 || !ctx->spares[ctx->pipe_depth - 2].prepared) {
    set_err(ctx, "no earlier hyperbatch in flight (needs a pipeline depth above 1 and two prepares)");
    return AGNES_ESTATE;
  }
  agnes_ctx::Spare& prev = ctx->spares[ctx->pipe_depth - 2];
  swap_hyperbatch_state(ctx, prev);
  const agnes_status rc = agnes_fetch_hyperbatch(ctx, out);
  swap_hyperbatch_state(ctx, prev);
  return rc;
}

agnes_status agnes_fetch_earlier_hyperbatch(agnes_ctx* ctx, int32_t ago,
                                            agnes_hyperbatch_view* out) {
  if (!ctx || !out) {
    set_err(ctx, "ctx and out must be non-NULL");
    return AGNES_EINVAL;
  }
  if (ago < 0 || ago >= ctx->pipe_depth) {
    set_err(ctx, "ago = %d outside [0, %d) (the pipeline depth)", ago, ctx->pipe_depth);
    return AGNES_EINVAL;
  }
  if (ago == 0) return agnes_fetch_hyperbatch(ctx, out);
  // spares[d - 2] holds the previous hyperbatch, spares[0] the oldest
  agnes_ctx::Spare& o = ctx->spares[ctx->pipe_depth - 1 - ago];
  if (!o.prepared) {
    set_err(ctx, "no hyperbatch %d prepares before the last one", ago);
    return AGNES_ESTATE;
  }
  swap_hyperbatch_state(ctx, o);
  const agnes_status rc = agnes_fetch_hyperbatch(ctx, out);
  swap_hyperbatch_state(ctx, o);
  return rc;
}

agnes_status agnes_wait_hyperbatches(agnes_ctx* ctx, void* cuda_stream) {
  if (!ctx) return AGNES_EINVAL;
  DeviceGuard dg(ctx->device);
  cudaStream_t st = (cudaStream_t)cuda_stream;
  if (ctx->done) CK(ctx, cudaStreamWaitEvent(st, ctx->done, 0));
  for (int i = 0; i + 1 < ctx->pipe_depth; ++i)
    if (ctx->spares[i].done) CK(ctx, cudaStreamWaitEvent(st, ctx->spares[i].done, 0));
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
  DeviceGuard dg(ctx->device);
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
  DeviceGuard dg(ctx->device);
  CK(ctx, cudaMemcpy(start_node, ctx->bt.start_node, sizeof(int32_t) * n, cudaMemcpyDeviceToHost));
  CK(ctx, cudaMemcpy(start_block, ctx->bt.start_block, sizeof(int32_t) * n,
                     cudaMemcpyDeviceToHost));
  return AGNES_OK;
}

agnes_status agnes_set_profiling(agnes_ctx* ctx, int32_t mode) {
  if (!ctx) return AGNES_EINVAL;
  if (mode != AGNES_PROFILE_OFF && mode != AGNES_PROFILE_PHASES && mode != AGNES_PROFILE_GATHER) {
    set_err(ctx, "profiling mode must be AGNES_PROFILE_OFF, _PHASES or _GATHER");
    return AGNES_EINVAL;
  }
  ctx->profiling = mode;
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
