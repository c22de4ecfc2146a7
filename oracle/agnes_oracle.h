/*
 * agnes_oracle.h -- plain single-threaded C oracle for AGNES hyperbatch
 * sampling + gathering (arXiv 2601.01473).
 *
 * TEST INFRASTRUCTURE ONLY.  This header and agnes_oracle.c exist to check
 * the CUDA path.  Only tests/, __graft_entry__.smoke() and bench.py's
 * cpu_baseline / reference legs may load or call them.  The product library
 * (libagnes.so) never includes, links or calls anything in oracle/, and the
 * oracle includes nothing from the product.
 *
 * What it computes is the plain per-minibatch definition of the method: the
 * block/hyperbatch organisation of Algorithm 1 (Sec. 3.3, Sec. 3.5) changes
 * the order in which work is done, never the sampled sets, so the oracle
 * samples each minibatch on its own, without blocks (Algorithm 1's
 * per-minibatch Sample and Gather calls).  Blocks appear only in the
 * blocks-touched statistics (Sec. 3.2 storage layer; Fig. 7's #I/O counts).
 *
 * All functions are reentrant (no global state) so a caller may run several
 * minibatches on separate threads.
 */
#ifndef AGNES_ORACLE_H
#define AGNES_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ORC_MAX_HOPS 8

/* Status codes (0 = ok). */
#define ORC_OK 0
#define ORC_EINVAL 1
#define ORC_ENOMEM 2

/* Graph in CSR form plus a row-major feature matrix, all in host memory.
 * offsets: N+1 entries of offsets_bits (32 or 64) bits; indices: E int32;
 * features: N rows of row_bytes bytes each (may be NULL if no gather). */
typedef struct {
  int64_t num_nodes;
  int64_t num_edges;
  const void* offsets;
  int32_t offsets_bits;
  const int32_t* indices;
  const uint8_t* features;
  int64_t row_bytes;
} orc_graph;

/* Result for one minibatch.  For hop h (0-based array index, hop number
 * h+1): dst_h = nodes[0 .. num_dst[h]), src_h = nodes[0 .. num_src[h]),
 * indptr[h] has num_dst[h]+1 entries, nbr[h] / col[h] have num_edges[h]
 * entries.  nodes holds src_K (num_nodes ids) and feats num_nodes rows. */
typedef struct {
  int32_t K;
  int64_t num_dst[ORC_MAX_HOPS];
  int64_t num_src[ORC_MAX_HOPS];
  int64_t num_edges[ORC_MAX_HOPS];
  int64_t* indptr[ORC_MAX_HOPS];
  int32_t* nbr[ORC_MAX_HOPS];
  int32_t* col[ORC_MAX_HOPS];
  int32_t* nodes;
  int64_t num_nodes;
  uint8_t* feats;
  int32_t* dst[ORC_MAX_HOPS]; /* dst_h (num_dst[h] ids) of every hop */
} orc_minibatch;

/* Which nodes form the next hop's frontier.
 * ORC_FRONTIER_SRC: dst_{h+1} = src_h = dst_h ++ new_h (every node reached so
 *   far, so eq. (1) has an embedding for every dst at every layer).
 * ORC_FRONTIER_SAMPLED: dst_{h+1} = N_out, the distinct ids sampled at hop h
 *   in ascending order (Algorithm 1 read literally: N_in <- N_out).
 * Blocks (src_h = dst_h ++ new_h, col into src_h) and the gathered src_{K-1}
 * are defined the same way in both. */
#define ORC_FRONTIER_SRC 0
#define ORC_FRONTIER_SAMPLED 1

/* Philox4x32 with 10 rounds (Salmon, Moraes, Dror, Shaw, SC'11). */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2],
                       uint32_t out[4]);

/* floor(a * b / 2^64), the high half of the full 128-bit product. */
uint64_t orc_mulhi64(uint64_t a, uint64_t b);

/* Positions (0-based offsets into v's adjacency list) of the neighbours
 * that node v samples at hop `hop` (1-based) of global minibatch g.  Writes
 * min(deg, k) positions to pos_out in slot order and returns that count. */
int64_t orc_sample_positions(uint64_t seed, uint64_t g, int32_t hop,
                             int32_t v, int64_t deg, int32_t k,
                             int64_t* pos_out);

/* Greedy packing of adjacency objects into fixed-size blocks (Sec. 3.2,
 * storage layer).  Writes node_block[v] (the block holding the start of v's
 * object) for all N nodes and returns the total block count (continuation
 * blocks of split objects included) in *num_blocks. */
int orc_build_adj_blocks(const orc_graph* g, int64_t block_bytes,
                         int32_t* node_block, int64_t* num_blocks);

/* Samples and gathers one minibatch (global id g).  targets: B distinct
 * node ids.  fanouts: K entries (fanouts[0] applies to the targets).
 * The frontier is ORC_FRONTIER_SRC. */
int orc_sample_minibatch(const orc_graph* g, const int32_t* targets,
                         int32_t B, const int32_t* fanouts, int32_t K,
                         uint64_t seed, uint64_t gid, int do_gather,
                         orc_minibatch* out);

/* The same with the frontier rule chosen by frontier_mode. */
int orc_sample_minibatch_mode(const orc_graph* g, const int32_t* targets,
                              int32_t B, const int32_t* fanouts, int32_t K,
                              uint64_t seed, uint64_t gid, int do_gather,
                              int32_t frontier_mode, orc_minibatch* out);

void orc_free_minibatch(orc_minibatch* mb);

/* Blocks-touched statistics for a hyperbatch of H already-sampled
 * minibatches: out[h] (h < K) = number of distinct adjacency blocks that
 * hold a node of dst_h (the frontier of hop h + 1) of any minibatch; out[K] = number of distinct
 * feature blocks (feat_rows_per_block rows each) that hold a node of src_K
 * of any minibatch. */
int orc_hyperbatch_stats(const orc_graph* g, const orc_minibatch* mbs,
                         int32_t H, int64_t adj_block_bytes,
                         int64_t feat_rows_per_block, int64_t* out);

#ifdef __cplusplus
}
#endif
#endif
