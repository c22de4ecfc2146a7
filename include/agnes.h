/*
 * agnes.h -- C ABI of libagnes.so: block-wise, hyperbatch-based multi-hop
 * neighbour sampling and feature gathering on one GB300 GPU (sm_103a), after
 * AGNES (arXiv 2601.01473).
 *
 * The operation (Algorithm 1, Sec. 3.5): given a graph's topology B_g and
 * features B_f cut into fixed-size blocks (Sec. 3.2, storage layer) and the
 * target nodes of a hyperbatch of H minibatches (Sec. 3.3), run K hops of
 * sampling -- each hop buckets the frontier by (block, minibatch) (the
 * bucket matrix Bck of Sec. 3.4 (3)), visits every non-empty block row once
 * for all minibatches, draws up to fanout[h] neighbours per frontier node
 * and unions the draws per minibatch -- then gather every sampled node's
 * feature row block by block (Algorithm 1's gathering loop).  The sampled
 * nodes N_s and gathered features F_g (Algorithm 1's outputs) stay in device
 * memory, one view per minibatch.
 *
 * Semantics fixed by this library where the paper is silent:
 *  - Sampling is uniform without replacement over a node's adjacency
 *    positions; a node with deg <= fanout takes all neighbours in CSR order;
 *    otherwise Floyd's algorithm with Philox4x32-10 draws keyed on
 *    key = (lo32 seed, hi32 seed), ctr = (v, (hop << 24) | slot,
 *    lo32 g, hi32 g), g = first_minibatch_id + j, hop = 1..K, and
 *    t = floor(((x1 << 32) | x0) * (J + 1) / 2^64).  Draws therefore depend
 *    on the global minibatch id, never on H, the block size or the order of
 *    work, and results are bit-exact and deterministic.
 *  - Per hop h of minibatch j: dst_h = the frontier, new_h = the ascending
 *    unique sampled ids not in dst_h, src_h = dst_h ++ new_h, and
 *    dst_{h+1} = src_h (hop 1's dst is the targets, in the caller's order).
 *    col[e] indexes the e-th sampled neighbour in src_h; edges are grouped by
 *    dst position (indptr) and in draw order within a dst.
 *  - Feature rows are copied byte for byte (fp32 / fp16 bit patterns,
 *    NaN payloads included).
 *
 * Conventions: every call returns an agnes_status and never throws; on
 * failure agnes_last_error(ctx) gives a message.  All work of a call is
 * enqueued on the caller's CUDA stream (NULL = the legacy default stream);
 * calls on one ctx must not overlap.  Pointers are host or device memory as
 * stated per argument; the library detects which with
 * cudaPointerGetAttributes where both are allowed.  A call that works on the
 * GPU makes the ctx's device current for its duration and restores the
 * calling thread's current device before it returns.
 */
#ifndef AGNES_H
#define AGNES_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define AGNES_MAX_HOPS 8
#define AGNES_MAX_PIPELINE_DEPTH 4 /* hyperbatches in flight (agnes_set_pipeline_depth) */
#define AGNES_MAX_FANOUT 65536

typedef enum {
  AGNES_OK = 0,
  AGNES_EINVAL = 1,   /* invalid argument or input data */
  AGNES_ERANGE = 2,   /* sizes overflow the library's index types */
  AGNES_ENOMEM = 3,   /* device or pinned host allocation failed */
  AGNES_ECUDA = 4,    /* a CUDA runtime call failed */
  AGNES_ESTATE = 5,   /* call out of order (e.g. fetch before prepare) */
  AGNES_ETIMEOUT = 6, /* a bounded wait ran out (on the host, or between CTAs of a kernel) */
  AGNES_EKERNEL = 7   /* a kernel reported an internal inconsistency */
} agnes_status;

typedef enum { AGNES_F32 = 0, AGNES_F16 = 1 } agnes_dtype;

typedef struct agnes_ctx agnes_ctx; /* opaque, owned by the library */

/* Graph description for agnes_load_graph (CSR + row-major features).
 *  num_nodes   N, 1 <= N < 2^31.
 *  num_edges   E = offsets[N] (offsets[0] must be 0).
 *  offsets     N+1 entries of offsets_bits (32 or 64) bits; host or device.
 *  indices     E int32 neighbour ids in [0, N); host or device.
 *  features    N x feat_dim elements of feat_dtype, row-major; host or
 *              device, or pinned host memory when features_on_host = 1.
 *  adj_block_bytes   size of a topology block (Sec. 3.2); >= 64.
 *  feat_block_bytes  size of a feature block; >= one feature row.
 * Host arrays are copied to device memory the library owns.  Device arrays
 * are borrowed: the caller keeps them alive and unchanged until
 * agnes_free.  With features_on_host = 1 the feature matrix stays in pinned
 * host memory (borrowed; 16-byte aligned, rows a multiple of 16 bytes) and
 * each hyperbatch reads what it needs over the host link, which stands in
 * for the SSD: whole feature blocks into device staging slots on a side
 * stream (feature_io = AGNES_FEATURE_IO_BLOCKS, the asynchronous block I/O
 * of Sec. 3.4 (4)), or only the requested rows (AGNES_FEATURE_IO_ROWS).
 * With topology_on_host = 1 the neighbour lists (indices, pinned host
 * memory, borrowed) stay on the host; offsets are still copied or borrowed
 * in device memory.  Each hop loads the topology blocks its frontier touches
 * into an HBM graph buffer of graph_buffer_bytes (a whole number of blocks,
 * at least the largest object), reusing resident blocks and evicting the
 * least recently used unpinned ones; a block stays pinned until the hop has
 * sampled all its requests (Sec. 3.4 (1)).  When a hop's blocks do not fit,
 * the hop runs in waves of blocks in ascending order.
 * With features_on_host = 1 and feature_cache_bytes > 0, an HBM feature
 * cache (Sec. 3.4 (2)) keeps the feature blocks whose cumulative request
 * count (rows gathered from them, over all hyperbatches so far) exceeds
 * feature_cache_threshold, hottest first, up to its capacity
 * (feature_cache_bytes / feature block size blocks).  The set is re-picked
 * after each hyperbatch; a newly admitted block is loaded into its cache
 * slot the next time a hyperbatch touches it and read in place from then on.
 * The cache holds whole feature blocks, the unit of host transfers. */
typedef struct {
  int64_t num_nodes;
  int64_t num_edges;
  const void* offsets;
  int32_t offsets_bits;
  const int32_t* indices;
  const void* features;
  int32_t feat_dtype; /* agnes_dtype */
  int64_t feat_dim;
  int32_t features_on_host;
  int64_t adj_block_bytes;
  int64_t feat_block_bytes;
  int32_t topology_on_host; /* 1: indices stay in pinned host memory (see below) */
  int64_t graph_buffer_bytes; /* topology_on_host: HBM graph buffer (blocks I/O; 0: whole
                                 topology) or topology cache (rows I/O; 0: none) */
  int64_t feature_cache_bytes;     /* features_on_host: HBM feature cache (0: none) */
  int64_t feature_cache_threshold; /* cumulative requests a block must exceed to be cached */
  int32_t feature_io;              /* features_on_host: AGNES_FEATURE_IO_BLOCKS or _ROWS */
  int32_t topology_io;             /* topology_on_host: AGNES_TOPOLOGY_IO_BLOCKS or _ROWS */
} agnes_graph_desc;

/* How host-resident neighbour lists reach the sampler (topology_on_host = 1).
 * BLOCKS: the blocks a hop's frontier touches are loaded whole into the HBM
 *   graph buffer (LRU + pinning, Sec. 3.4 (1)); 0, the default.
 * ROWS: the sampler reads each sampled neighbour entry in place from pinned
 *   host memory over the host link.  Not in the paper, for the reason given
 *   for feature rows.  With graph_buffer_bytes > 0 the buffer is a topology
 *   cache instead: the block runs (a block start and its continuation
 *   blocks) with the most frontier requests since load are kept in it,
 *   hottest first, up to its capacity, in the spirit of the count-based
 *   feature cache of Sec. 3.4 (2); the sampler reads a cached block from HBM
 *   and any other in place.  The set is picked before the 2nd hyperbatch and
 *   re-picked every 8 hyperbatches after; a prepare that re-picks first waits
 *   for the previous hyperbatch. */
#define AGNES_TOPOLOGY_IO_BLOCKS 0
#define AGNES_TOPOLOGY_IO_ROWS 1

/* How host-resident features reach the gather (features_on_host = 1).
 * BLOCKS: every touched feature block is loaded whole into HBM, batch by
 *   batch, overlapped with the gather (the block-wise I/O of Sec. 3.3 and the
 *   asynchronous I/O of Sec. 3.4 (4)); 0, the default.
 * ROWS: only requested rows cross the host link, read in place from pinned
 *   host memory by the GPU.  Without a feature cache, each distinct requested
 *   row of the hyperbatch crosses once into an HBM staging area that serves
 *   every request; with a cache, every row is read where its block is (cache
 *   slot or host memory), since the rows several minibatches request are
 *   then mostly in the cache.  Not in the paper: its storage is an SSD, where small
 *   reads are slow; a cache-coherent host link serves row-sized reads at the
 *   rate of bulk copies. */
#define AGNES_FEATURE_IO_BLOCKS 0
#define AGNES_FEATURE_IO_ROWS 1

/* Loads a graph on `device` and builds its block tables: the object index
 * table T^g_obj of Sec. 3.2 (greedy in-order packing of objects of
 * offsets_bits/8 + 4*deg bytes into adj_block_bytes blocks; an object larger
 * than a block starts a fresh block and spans ceil(size/block) blocks) and
 * the feature blocks (feat_block_bytes / row_bytes rows each).  Enqueued on
 * cuda_stream and synchronised before return.  *out receives a new ctx (NULL
 * on failure).  Errors: EINVAL (bad desc), ERANGE, ENOMEM, ECUDA. */
agnes_status agnes_load_graph(const agnes_graph_desc* desc, int device, void* cuda_stream,
                              agnes_ctx** out);

/* Samples K hops and gathers features for a hyperbatch of H minibatches of
 * B targets each (Algorithm 1).
 *  targets   H*B int32 node ids, row j = minibatch j's targets (distinct
 *            within a row); host or device memory.  Host memory is copied
 *            inside the call (pinned memory makes that copy asynchronous).
 *  fanouts   K host int32 values, fanouts[0] for the targets' hop;
 *            1 <= fanouts[h] <= AGNES_MAX_FANOUT, 1 <= K <= AGNES_MAX_HOPS.
 *            A hop with a fanout above 1024 also uses ctx-owned device
 *            memory for the sampler's per-warp sets of chosen positions
 *            (at most 1 GiB, allocated with the workspace).
 *  seed, first_minibatch_id  key the random draws (see above).
 * Stream-ordered: returns once the work is enqueued, after the ctx's previous
 * prepare (on whatever stream) and before anything later on cuda_stream.
 * Issued while cuda_stream is being captured into the caller's own CUDA
 * graph, the work is recorded into that graph instead of run: fetch and
 * stats describe it only once the caller has launched the graph and waited
 * for it, the caller orders those launches with the ctx's other prepares,
 * and no phase times are recorded.  Element-wise checks of
 * targets (range, distinctness) run on the device and are reported by the
 * next agnes_fetch_minibatch / agnes_hyperbatch_stats call as EINVAL.
 * Errors here: EINVAL (bad scalar args), ERANGE (H * capacity >= 2^31 output
 * rows, or H * the graph's tiles >= 2^31 bucket cells), ENOMEM, ECUDA. */
agnes_status agnes_prepare_hyperbatch(agnes_ctx* ctx, const int32_t* targets, int32_t H,
                                      int32_t B, const int32_t* fanouts, int32_t K,
                                      uint64_t seed, uint64_t first_minibatch_id,
                                      void* cuda_stream);

/* Which nodes form each next hop's frontier (set per ctx; takes effect at
 * the next agnes_prepare_hyperbatch).
 * AGNES_FRONTIER_SRC (default): dst_{h+1} = src_h = dst_h ++ new_h, every
 *   node reached so far, so the layer of eq. (1) over each hop has an input
 *   row for each of its src nodes from the layer below.
 * AGNES_FRONTIER_SAMPLED: dst_{h+1} = N_out, the distinct ids sampled at hop
 *   h in ascending order (Algorithm 1's frontier update N_in <- N_out read
 *   literally).  Only the frontier update is literal: the output is still
 *   the per-hop blocks and the rows of the last hop's src list (below), not
 *   Algorithm 1's N_s, the union of every hop's N_out, which would drop the
 *   rows the lower hops' blocks index.
 * In both, hop h's block has src_h = dst_h ++ new_h (new_h = the sampled ids
 * not in dst_h, ascending) and col indexes src_h; the gathered rows are
 * src_{K-1}.  Errors: EINVAL. */
#define AGNES_FRONTIER_SRC 0
#define AGNES_FRONTIER_SAMPLED 1
agnes_status agnes_set_frontier_mode(agnes_ctx* ctx, int32_t mode);

/* How agnes_prepare_hyperbatch issues its work when features and topology
 * are resident in HBM (set per ctx; takes effect at the next prepare).
 * AGNES_LAUNCH_DIRECT: every call launches the sequence (memsets, ~60
 *   kernels, the size read-back) on the caller's stream.
 * AGNES_LAUNCH_GRAPH: the sequence is captured into a CUDA graph on a
 *   private stream the first time a hyperbatch shape is seen (H, B, fanouts,
 *   frontier mode, profiling) and replayed as one graph launch on the
 *   caller's stream for every later hyperbatch of that shape; the targets
 *   copy and the sampling key {seed, first_minibatch_id} are written to
 *   device memory ahead of it.
 * AGNES_LAUNCH_GRAPH_PDL (default): as AGNES_LAUNCH_GRAPH, with each link of
 *   the graph's kernel chain (one predecessor, one successor) made
 *   programmatic (programmatic dependent launch: a kernel is launched once
 *   every block of the previous one has exited, and first waits for its
 *   writes to become visible), so each launch overlaps the previous kernel's
 *   completion.
 * In every mode, work off the critical chain (each hop's new-id scan and col
 * fix-up, the touched-block statistics) runs on a side stream the ctx owns,
 * forked from and joined back into the caller's stream within the call's
 * work.  Results are identical in every mode.  A caller stream that is itself being
 * captured, and the host-resident modes (whose calls read sizes back
 * mid-sequence), always take the direct path.  Errors: EINVAL. */
#define AGNES_LAUNCH_DIRECT 0
#define AGNES_LAUNCH_GRAPH 1
#define AGNES_LAUNCH_GRAPH_PDL 2
agnes_status agnes_set_launch_mode(agnes_ctx* ctx, int32_t mode);

/* View of minibatch j of the last prepared hyperbatch.  Per hop h (0-based
 * index, hop number h+1): the bipartite block has num_dst[h] dst nodes and
 * num_src[h] src nodes, dst_h being the first num_dst[h] of src_h (with the
 * default frontier, both are prefixes of nodes); indptr[h] (num_dst[h]+1 int64, device) groups
 * the num_edges[h] edges by dst; col[h] (num_edges[h] int32, device) gives
 * each edge's src index.  nodes (num_nodes int32, device) = src_K in global
 * ids; feats (num_nodes x feat_dim of feat_dtype, device, row-major) their
 * gathered rows.  All pointers are owned by ctx and stay valid until the
 * next agnes_prepare_hyperbatch or agnes_free. */
typedef struct {
  int32_t K;
  int64_t num_dst[AGNES_MAX_HOPS];
  int64_t num_src[AGNES_MAX_HOPS];
  int64_t num_edges[AGNES_MAX_HOPS];
  const int64_t* indptr[AGNES_MAX_HOPS];
  const int32_t* col[AGNES_MAX_HOPS];
  const int32_t* nodes;
  int64_t num_nodes;
  const void* feats;
  int32_t feat_dtype;
  int64_t feat_dim;
} agnes_minibatch_view;

/* Fills *out for minibatch j (0 <= j < H).  The first fetch after a prepare
 * waits for that hyperbatch's work (host-side, on an event) and reads its
 * sizes back once.  Errors: ESTATE (no hyperbatch), EINVAL (bad j, or bad
 * targets found on the device), ECUDA. */
agnes_status agnes_fetch_minibatch(agnes_ctx* ctx, int32_t j, agnes_minibatch_view* out);

/* All minibatches of the last hyperbatch at once, for callers that consume
 * the whole hyperbatch (one wait and one size read-back for all H views).
 * Minibatch j's arrays start at base + j * stride (elements), with the sizes
 * of agnes_fetch_minibatch:
 *   indptr[h] + j*indptr_stride[h]   num_dst = dst_size[h*H + j] (+1 entries)
 *   col[h] + j*col_stride[h]         num_edges = edges[h*H + j]
 *   nodes + j*nodes_stride           num_nodes = node_size[K*H + j]
 *   feats + j*feats_stride_rows*row_bytes
 * node_size[h*H + j] is |dst_h| of minibatch j for h < K (node_size[0..H)
 * = B) and num_nodes = |src_{K-1}| for h = K; src_size[h*H + j] is |src_h|
 * (equal to node_size[(h+1)*H + j] with the default frontier); edges is
 * K x H.  node_size, src_size and edges are host memory owned by ctx.  Everything stays valid until the next prepare or
 * free.  Errors as agnes_fetch_minibatch. */
typedef struct {
  int32_t K, H;
  const int64_t* indptr[AGNES_MAX_HOPS];
  int64_t indptr_stride[AGNES_MAX_HOPS];
  const int32_t* col[AGNES_MAX_HOPS];
  int64_t col_stride[AGNES_MAX_HOPS];
  const int32_t* nodes;
  int64_t nodes_stride;
  const void* feats;
  int64_t feats_stride_rows;
  int32_t feat_dtype;
  int64_t feat_dim;
  const int32_t* node_size;
  const int32_t* edges;
  const int32_t* src_size;  /* K x H: |src_h| of minibatch j at h*H + j */
} agnes_hyperbatch_view;
agnes_status agnes_fetch_hyperbatch(agnes_ctx* ctx, agnes_hyperbatch_view* out);

/* Hyperbatches in flight.  depth 1 (the default): each prepare is ordered on
 * the caller's stream as described at agnes_prepare_hyperbatch.  depth d in
 * 2 .. AGNES_MAX_PIPELINE_DEPTH: the ctx keeps d workspaces (d times the
 * device memory of one) and d sets of internal streams, and consecutive
 * prepares use the sets in turn, each on its own internal stream that starts
 * when the caller's stream reaches the call and once the set's previous
 * hyperbatch (d prepares earlier) is done; the caller's stream is not made to
 * wait for the hyperbatch, so consecutive hyperbatches overlap (Sec. 3.4 (4):
 * one stage's latency hidden behind another's work).  Then: fetch, stats and
 * counters wait for and describe the last prepared hyperbatch (host side, as
 * before); a stream that consumes the views on the device must first be
 * ordered with agnes_wait_hyperbatches; views stay valid until the d-th
 * prepare after the one they come from.  depth > 1 needs the graph resident
 * in device memory (no features_on_host, no topology_on_host); a prepare
 * issued while the caller's stream is being captured runs as at depth 1.
 * The call waits for the device; changing the depth releases the spare sets,
 * so only the last hyperbatch's views survive it.  Errors: EINVAL, ECUDA. */
agnes_status agnes_set_pipeline_depth(agnes_ctx* ctx, int32_t depth);

/* At depth > 1: the views of the hyperbatch prepared before the last one
 * (waiting for it like agnes_fetch_hyperbatch), so a caller can take one
 * hyperbatch's results while the next is being prepared.  They stay valid
 * until the (depth - 1)-th prepare after this call.  Errors: EINVAL, ESTATE
 * (depth 1, or fewer than two prepares), ECUDA, and what
 * agnes_fetch_hyperbatch reports. */
agnes_status agnes_fetch_previous_hyperbatch(agnes_ctx* ctx, agnes_hyperbatch_view* out);

/* At depth d: the views of the hyperbatch prepared `ago` prepares before the
 * last one, 0 <= ago < d (0: as agnes_fetch_hyperbatch; 1: as
 * agnes_fetch_previous_hyperbatch), waiting for it, so a caller can take the
 * oldest hyperbatch still held while the later ones run.  They stay valid
 * until the (d - ago)-th prepare after this call.  Errors: EINVAL (ago out
 * of range), ESTATE (fewer than ago + 1 prepares at this depth), ECUDA, and
 * what agnes_fetch_hyperbatch reports. */
agnes_status agnes_fetch_earlier_hyperbatch(agnes_ctx* ctx, int32_t ago,
                                            agnes_hyperbatch_view* out);

/* Makes cuda_stream wait (on the device) for every hyperbatch prepared and
 * still in flight on the ctx: the last depth prepares.  Errors: EINVAL,
 * ECUDA. */
agnes_status agnes_wait_hyperbatches(agnes_ctx* ctx, void* cuda_stream);

/* Blocks touched by the last hyperbatch (the block-wise I/Os of Sec. 3.3 and
 * Fig. 7): out[h] for h < K = distinct topology blocks holding a node of
 * some minibatch's hop-(h+1) frontier; out[K] = distinct feature blocks
 * holding a gathered node.  out has K+1 host entries.  Waits like fetch. */
agnes_status agnes_hyperbatch_stats(agnes_ctx* ctx, int64_t* out);

/* Whole-hyperbatch totals of the last hyperbatch, for byte accounting.
 * Waits like fetch. */
typedef struct {
  int32_t K;
  int64_t frontier[AGNES_MAX_HOPS]; /* sum over minibatches of num_dst[h] */
  int64_t edges[AGNES_MAX_HOPS];    /* sum over minibatches of num_edges[h] */
  int64_t rows;                     /* sum over minibatches of num_nodes */
  int64_t distinct_rows;            /* distinct node ids among all gathered rows */
  int64_t row_bytes;
  int64_t streamed_bytes;           /* features_on_host: bytes read over the host link
                                       (row mode: distinct rows without a cache, every
                                       request of an uncached block with one; plus
                                       blocks loaded into the cache) */
  int64_t streamed_blocks;          /* features_on_host: touched feature blocks not
                                       served by the feature cache */
  /* the rest are totals since agnes_load_graph, not per hyperbatch */
  int64_t topo_loaded_blocks;       /* topology_on_host: blocks copied into the graph buffer
                                       or the topology cache */
  int64_t topo_loaded_bytes;
  int64_t topo_hit_blocks;          /* needed blocks already resident (blocks I/O) */
  int64_t topo_waves;               /* fill launches over all hops */
  int64_t fcache_hit_blocks;        /* feature blocks read in place from the feature cache */
  int64_t fcache_loaded_blocks;     /* feature blocks copied into the feature cache */
  int64_t graph_captures;           /* launch sequences captured (agnes_set_launch_mode) */
  int64_t graph_launches;           /* prepares issued as one graph launch */
  int64_t graph_programmatic_edges; /* programmatic kernel edges of the current graph */
  int64_t topo_cached_requests;     /* rows I/O with a topology cache: frontier entries
                                       whose topology block was cached */
} agnes_counters;
agnes_status agnes_hyperbatch_counters(agnes_ctx* ctx, agnes_counters* out);

/* Static facts about the loaded graph.  adj_blocks counts continuation
 * blocks of split objects; tiles is the number of (topology block x
 * feature block x 4096-id chunk) cells the buckets are kept in. */
typedef struct {
  int64_t num_nodes, num_edges;
  int64_t adj_blocks, adj_block_starts, feat_blocks, feat_rows_per_block, tiles;
  int64_t row_bytes;
} agnes_graph_info;
agnes_status agnes_get_graph_info(agnes_ctx* ctx, agnes_graph_info* out);

/* Copies the object index table to host memory: for each of the first
 * min(cap, adj_block_starts) block starts, the first node whose object
 * starts there (start_node) and that block's index (start_block).
 * Continuation blocks of a split object are implied by the gaps between
 * consecutive start_block values. */
agnes_status agnes_copy_adj_blocks(agnes_ctx* ctx, int32_t* start_node, int32_t* start_block,
                                   int64_t cap);

/* Optional timing of later prepares with CUDA events on the caller's stream
 * (off by default; the events of the last 64 prepares are kept).
 * AGNES_PROFILE_PHASES: agnes_phase_times writes, in order, [0] bucketing of
 *   the targets, then per hop h (3 each): [1+3h] count+scan, [2+3h]
 *   sampling, [3+3h] dedup+relabel, then [1+3K] gather.
 * AGNES_PROFILE_GATHER: only [0] the gather.  Each event splits the launch
 *   sequence at that point (it is a dependency of what follows), so fewer
 *   events cost less: two instead of 3K + 3.
 * agnes_phase_times writes up to n milliseconds of the prepare issued `ago`
 * calls before the latest one (0 = the latest, < 64); *n_out receives the
 * count (0 if that prepare was not profiled).  Waits for the latest prepare
 * like fetch.  Errors: EINVAL (mode unknown, ago out of range). */
#define AGNES_PROFILE_OFF 0
#define AGNES_PROFILE_PHASES 1
#define AGNES_PROFILE_GATHER 2
agnes_status agnes_set_profiling(agnes_ctx* ctx, int32_t mode);
agnes_status agnes_phase_times(agnes_ctx* ctx, int32_t ago, float* ms, int32_t n,
                               int32_t* n_out);

/* A GraphSAGE-mean layer over hop `hop` of every minibatch of the last
 * hyperbatch: the consumer of the prepared blocks.  It is an instance of
 * eq. (1) (Sec. 3.1), with the mean of the in-neighbours' rows as the
 * aggregation and a fully connected layer with ReLU as the update:
 *   out_i = ReLU(W_self x_i + W_neigh mean_{e in row i} x_{col[e]} + b)
 * for every dst row i of the hop (dst_h is a prefix of src_h, so x_i is row
 * i of x).  Layers stack from the outermost hop in: hop K-1 takes the
 * gathered features (x = feats of agnes_fetch_hyperbatch, x_stride_rows =
 * feats_stride_rows) and its output rows are src_{K-2}, the input of hop K-2.
 *  x      device, minibatch j's src_h rows at x + (j*x_stride_rows + r)*d_in
 *         elements of x_dtype (AGNES_F32 or AGNES_F16); x_stride_rows >= the
 *         largest |src_h|.
 *  w      device, d_out x 2*d_in IEEE fp16, row-major: columns [0, d_in)
 *         multiply x_i (W_self), [d_in, 2*d_in) the mean (W_neigh).
 *  bias   device, d_out floats, or NULL for none.
 *  out    device, minibatch j's dst_h rows at out + (j*out_stride_rows + i)*
 *         d_out elements of out_dtype; out_stride_rows >= the largest |dst_h|.
 * Arithmetic: the mean is summed and divided in fp32, the update's inputs
 * are rounded to fp16, and the products are accumulated in fp32 on the
 * tensor cores (tcgen05).  d_in is a multiple of 8, d_out a multiple of 32
 * in [32, 256], and W plus one 128-row tile of [x_i | mean_i] must fit
 * shared memory: 512*d_in + 4*d_in*d_out + 128 <= AGNES_SAGE_MAX_SMEM bytes
 * (ERANGE otherwise).  Scratch: the layer keeps [x_i | mean_i] of every dst
 * row (4*d_in bytes each) in device memory owned by ctx.  x, w and out are 16-byte aligned.  Waits for the hyperbatch
 * like agnes_fetch_hyperbatch, runs on cuda_stream and waits for it.
 * Errors: EINVAL, ERANGE, ESTATE, ECUDA, ETIMEOUT (a tensor-core completion
 * wait ran out; the layer's output is then undefined). */
#define AGNES_SAGE_MAX_SMEM 232448
agnes_status agnes_sage_mean_layer(agnes_ctx* ctx, int32_t hop, const void* x, int32_t x_dtype,
                                   int64_t x_stride_rows, int64_t d_in, const void* w,
                                   const float* bias, int32_t d_out, void* out,
                                   int32_t out_dtype, int64_t out_stride_rows,
                                   void* cuda_stream);

/* Allocation-free variant of one step of the path: for a node list (for
 * example one minibatch's frontier), the per-node edge counts of one hop's
 * sampling, min(deg(v), fanout), and their prefix sum -- the indptr that
 * agnes_prepare_hyperbatch computes for each hop.  It exists for callers
 * that must not allocate device memory: a latency-critical loop cannot
 * afford the device-wide synchronisation cudaFree implies, and a process
 * whose device memory is all reserved by another allocator (a framework's
 * caching pool) may find cudaMalloc failing.  The paper has no counterpart;
 * this is a library convenience.
 *  nodes   n int32 node ids in [0, N), device memory.
 *  indptr  n+1 int64, device memory: indptr[0] = 0,
 *          indptr[i+1] = indptr[i] + min(deg(nodes[i]), fanout).
 *  n       0 <= n <= AGNES_NOALLOC_MAX_NODES, else ERANGE.
 *  fanout  1 <= fanout <= AGNES_MAX_FANOUT.
 * Its scratch (64 KiB: per-chunk partial sums and an error word) is a
 * static device array that every GPU loading the library holds until the
 * process exits; nothing is allocated per call.  Each call looks up that
 * array's device address on the ctx's device (a host-side query).  All calls
 * on a device share the array: calls that overlap on the GPU race and must be
 * serialised by the caller.  The call enqueues its work on cuda_stream and
 * then synchronises that stream (to report node ids outside [0, N) as
 * EINVAL), so it must not be made while cuda_stream is being captured into a
 * CUDA graph.  Errors: EINVAL, ERANGE, ECUDA. */
#define AGNES_NOALLOC_MAX_NODES (1LL << 24)
agnes_status agnes_hop_indptr_noalloc(agnes_ctx* ctx, const int32_t* nodes, int64_t n,
                                      int32_t fanout, int64_t* indptr, void* cuda_stream);

/* Releases everything the ctx owns (after synchronising its streams). */
agnes_status agnes_free(agnes_ctx* ctx);

const char* agnes_status_string(agnes_status s);
const char* agnes_last_error(agnes_ctx* ctx); /* "" when none; ctx may be NULL */

#ifdef __cplusplus
}
#endif
#endif
