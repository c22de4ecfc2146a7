/*
 * agnes_oracle.c -- plain single-threaded C oracle for AGNES hyperbatch
 * sampling + gathering (arXiv 2601.01473).
 *
 * TEST INFRASTRUCTURE ONLY: see agnes_oracle.h.  Written for obviousness,
 * not speed; nothing here is shared with the CUDA path.
 *
 * Per minibatch g (Algorithm 1's Sample(j, ...) and Gather(j, ...), Sec. 3.5):
 *   dst_1 = targets_g
 *   for hop h = 1..K:
 *     for each v in dst_h: draw up to k_h neighbour positions of v without
 *       replacement (all of them when deg(v) <= k_h), keyed on
 *       (seed, g, h, v, slot) so the draw does not depend on which block or
 *       hyperbatch the request arrives in;
 *     new_h = ascending unique sampled ids that are not in dst_h   (the
 *       union N_out <- N_out u Sample(...) of Algorithm 1)
 *     src_h = dst_h ++ new_h; col[e] = index of the e-th neighbour in src_h
 *     dst_{h+1} = src_h
 *   feats = features[src_K]  (Gather)
 * Where the paper is silent this file takes these readings: sampling is
 * without replacement over adjacency positions, dst is kept as a prefix of
 * src, new nodes are in ascending id order, Philox is keyed as stated above,
 * and blocks are packed greedily in id order.  Each is a choice the paper
 * leaves open, not a result it fixes.
 */
#include "agnes_oracle.h"

#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------------
 * Philox4x32-10, from its published definition (Salmon et al., "Parallel
 * random numbers: as easy as 1, 2, 3", SC'11): ten rounds of a
 * multiply-xor S-box on a 4-word counter, with a 2-word key bumped by the
 * Weyl constants between rounds.
 * ------------------------------------------------------------------- */
#define ORC_PHILOX_M0 0xD2511F53u
#define ORC_PHILOX_M1 0xCD9E8D57u
#define ORC_PHILOX_W0 0x9E3779B9u
#define ORC_PHILOX_W1 0xBB67AE85u

void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2],
                       uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += ORC_PHILOX_W0;
      k1 += ORC_PHILOX_W1;
    }
    uint64_t p0 = (uint64_t)ORC_PHILOX_M0 * (uint64_t)c0;
    uint64_t p1 = (uint64_t)ORC_PHILOX_M1 * (uint64_t)c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    uint32_t n3 = lo0;
    c0 = n0;
    c1 = n1;
    c2 = n2;
    c3 = n3;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

uint64_t orc_mulhi64(uint64_t a, uint64_t b) {
  unsigned __int128 p = (unsigned __int128)a * (unsigned __int128)b;
  return (uint64_t)(p >> 64);
}

/* ---------------------------------------------------------------------
 * Uniform sampling without replacement of min(deg, k) positions out of
 * deg (the random subset of neighbours of Sec. 3.1).  deg <= k takes every
 * position in order.  Otherwise Floyd's algorithm (Bentley & Floyd,
 * "Programming pearls: a sample of brilliance", CACM 1987): for slot
 * s = 0..k-1 with J = deg-k+s, draw t uniform in [0, J]; keep t unless it
 * was already chosen, in which case keep J.
 * The draw for (seed, g, hop, v, s) is Philox4x32-10 with
 *   key = (lo32(seed), hi32(seed)),
 *   ctr = (v, (hop << 24) | s, lo32(g), hi32(g)),
 * r = (x1 << 32) | x0, and t = floor(r * (J+1) / 2^64).
 * ------------------------------------------------------------------- */
int64_t orc_sample_positions(uint64_t seed, uint64_t g, int32_t hop,
                             int32_t v, int64_t deg, int32_t k,
                             int64_t* pos_out) {
  if (deg <= (int64_t)k) {
    for (int64_t i = 0; i < deg; ++i) pos_out[i] = i;
    return deg;
  }
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  for (int32_t s = 0; s < k; ++s) {
    int64_t J = deg - (int64_t)k + s;
    uint32_t ctr[4] = {(uint32_t)v, ((uint32_t)hop << 24) | (uint32_t)s,
                       (uint32_t)g, (uint32_t)(g >> 32)};
    uint32_t x[4];
    orc_philox4x32_10(ctr, key, x);
    uint64_t r = ((uint64_t)x[1] << 32) | (uint64_t)x[0];
    int64_t t = (int64_t)orc_mulhi64(r, (uint64_t)(J + 1));
    int seen = 0;
    for (int32_t q = 0; q < s; ++q) {
      if (pos_out[q] == t) {
        seen = 1;
        break;
      }
    }
    pos_out[s] = seen ? J : t;
  }
  return k;
}

/* ---------------------------------------------------------------------
 * CSR helpers.
 * ------------------------------------------------------------------- */
static int64_t orc_offset(const orc_graph* g, int64_t i) {
  if (g->offsets_bits == 32) return (int64_t)((const int32_t*)g->offsets)[i];
  return ((const int64_t*)g->offsets)[i];
}

static int orc_check_graph(const orc_graph* g) {
  if (!g || g->num_nodes < 0 || g->num_edges < 0) return ORC_EINVAL;
  if (g->offsets_bits != 32 && g->offsets_bits != 64) return ORC_EINVAL;
  if (g->num_nodes > 0 && (!g->offsets || !g->indices)) return ORC_EINVAL;
  return ORC_OK;
}

/* ---------------------------------------------------------------------
 * Storage-layer blocks for the topology (Sec. 3.2): objects (a node's
 * offset header plus its 4-byte neighbour ids) are laid out in ascending
 * node id.  A block is filled greedily; an object that does not fit in the
 * rest of the current block starts the next block.  An object larger than
 * a block starts a fresh block and is split over ceil(size / block) blocks;
 * the next object starts after them.  The header is one offset
 * (offsets_bits / 8 bytes).
 * ------------------------------------------------------------------- */
int orc_build_adj_blocks(const orc_graph* g, int64_t block_bytes,
                         int32_t* node_block, int64_t* num_blocks) {
  if (orc_check_graph(g) != ORC_OK || block_bytes <= 0 || !num_blocks)
    return ORC_EINVAL;
  int64_t hdr = g->offsets_bits / 8;
  int64_t b = 0, used = 0;
  for (int64_t v = 0; v < g->num_nodes; ++v) {
    int64_t deg = orc_offset(g, v + 1) - orc_offset(g, v);
    int64_t size = hdr + 4 * deg;
    if (size > block_bytes) {
      if (used > 0) {
        b += 1;
        used = 0;
      }
      node_block[v] = (int32_t)b;
      b += (size + block_bytes - 1) / block_bytes;
      used = 0;
    } else {
      if (used + size > block_bytes) {
        b += 1;
        used = 0;
      }
      node_block[v] = (int32_t)b;
      used += size;
    }
  }
  *num_blocks = b + (used > 0 ? 1 : 0);
  return ORC_OK;
}

/* ---------------------------------------------------------------------
 * Per-minibatch sampling and gathering.
 * ------------------------------------------------------------------- */
static int orc_cmp_i32(const void* a, const void* b) {
  int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
  return (x > y) - (x < y);
}

typedef struct {
  int32_t id;
  int32_t pos;
} orc_idpos;

static int orc_cmp_idpos(const void* a, const void* b) {
  int32_t x = ((const orc_idpos*)a)->id, y = ((const orc_idpos*)b)->id;
  return (x > y) - (x < y);
}

/* Index of key in sorted a[0..n), or -1. */
static int64_t orc_find_i32(const int32_t* a, int64_t n, int32_t key) {
  int64_t lo = 0, hi = n;
  while (lo < hi) {
    int64_t mid = lo + (hi - lo) / 2;
    if (a[mid] < key)
      lo = mid + 1;
    else
      hi = mid;
  }
  return (lo < n && a[lo] == key) ? lo : -1;
}

static int64_t orc_find_idpos(const orc_idpos* a, int64_t n, int32_t key) {
  int64_t lo = 0, hi = n;
  while (lo < hi) {
    int64_t mid = lo + (hi - lo) / 2;
    if (a[mid].id < key)
      lo = mid + 1;
    else
      hi = mid;
  }
  return (lo < n && a[lo].id == key) ? lo : -1;
}

void orc_free_minibatch(orc_minibatch* mb) {
  if (!mb) return;
  for (int h = 0; h < ORC_MAX_HOPS; ++h) {
    free(mb->indptr[h]);
    free(mb->nbr[h]);
    free(mb->col[h]);
    free(mb->dst[h]);
    mb->indptr[h] = NULL;
    mb->nbr[h] = NULL;
    mb->col[h] = NULL;
    mb->dst[h] = NULL;
  }
  free(mb->nodes);
  free(mb->feats);
  mb->nodes = NULL;
  mb->feats = NULL;
}

int orc_sample_minibatch(const orc_graph* g, const int32_t* targets,
                         int32_t B, const int32_t* fanouts, int32_t K,
                         uint64_t seed, uint64_t gid, int do_gather,
                         orc_minibatch* out) {
  return orc_sample_minibatch_mode(g, targets, B, fanouts, K, seed, gid, do_gather,
                                   ORC_FRONTIER_SRC, out);
}

int orc_sample_minibatch_mode(const orc_graph* g, const int32_t* targets,
                              int32_t B, const int32_t* fanouts, int32_t K,
                              uint64_t seed, uint64_t gid, int do_gather,
                              int32_t frontier_mode, orc_minibatch* out) {
  if (orc_check_graph(g) != ORC_OK || !out || !fanouts || B < 0 || K < 1 ||
      K > ORC_MAX_HOPS || (B > 0 && !targets) ||
      (frontier_mode != ORC_FRONTIER_SRC && frontier_mode != ORC_FRONTIER_SAMPLED))
    return ORC_EINVAL;
  memset(out, 0, sizeof(*out));
  out->K = K;
  for (int h = 0; h < K; ++h)
    if (fanouts[h] < 1 || fanouts[h] > (1 << 16)) return ORC_EINVAL;
  for (int32_t i = 0; i < B; ++i)
    if (targets[i] < 0 || (int64_t)targets[i] >= g->num_nodes)
      return ORC_EINVAL;

  int rc = ORC_ENOMEM;
  int32_t* nodes = (int32_t*)malloc(sizeof(int32_t) * (size_t)(B > 0 ? B : 1));
  if (!nodes) return ORC_ENOMEM;
  memcpy(nodes, targets, sizeof(int32_t) * (size_t)B);
  int64_t n_nodes = B;

  /* Targets must be distinct within a minibatch. */
  {
    int32_t* chk = (int32_t*)malloc(sizeof(int32_t) * (size_t)(B > 0 ? B : 1));
    if (!chk) goto fail;
    memcpy(chk, targets, sizeof(int32_t) * (size_t)B);
    qsort(chk, (size_t)B, sizeof(int32_t), orc_cmp_i32);
    for (int32_t i = 1; i < B; ++i) {
      if (chk[i] == chk[i - 1]) {
        free(chk);
        rc = ORC_EINVAL;
        goto fail;
      }
    }
    free(chk);
  }

  for (int32_t h = 0; h < K; ++h) {
    const int32_t hop = h + 1;
    const int32_t k = fanouts[h];
    const int64_t nd = n_nodes; /* dst_h = nodes[0 .. nd) */
    out->num_dst[h] = nd;
    out->dst[h] = (int32_t*)malloc(sizeof(int32_t) * (size_t)(nd > 0 ? nd : 1));
    if (!out->dst[h]) goto fail;
    memcpy(out->dst[h], nodes, sizeof(int32_t) * (size_t)nd);

    /* Sample: indptr over dst positions, neighbour ids in slot order. */
    int64_t* indptr = (int64_t*)malloc(sizeof(int64_t) * (size_t)(nd + 1));
    if (!indptr) goto fail;
    out->indptr[h] = indptr;
    indptr[0] = 0;
    for (int64_t i = 0; i < nd; ++i) {
      int32_t v = nodes[i];
      int64_t deg = orc_offset(g, v + 1) - orc_offset(g, v);
      indptr[i + 1] = indptr[i] + (deg < k ? deg : k);
    }
    const int64_t ne = indptr[nd];
    out->num_edges[h] = ne;
    int32_t* nbr = (int32_t*)malloc(sizeof(int32_t) * (size_t)(ne > 0 ? ne : 1));
    int64_t* pos = (int64_t*)malloc(sizeof(int64_t) * (size_t)k);
    if (!nbr || !pos) {
      free(nbr);
      free(pos);
      goto fail;
    }
    out->nbr[h] = nbr;
    for (int64_t i = 0; i < nd; ++i) {
      int32_t v = nodes[i];
      int64_t base = orc_offset(g, v);
      int64_t deg = orc_offset(g, v + 1) - base;
      int64_t c = orc_sample_positions(seed, gid, hop, v, deg, k, pos);
      for (int64_t s = 0; s < c; ++s) nbr[indptr[i] + s] = g->indices[base + pos[s]];
    }
    free(pos);

    /* Union: new_h = sorted unique sampled ids that are not in dst_h. */
    orc_idpos* dsorted =
        (orc_idpos*)malloc(sizeof(orc_idpos) * (size_t)(nd > 0 ? nd : 1));
    int32_t* uniq = (int32_t*)malloc(sizeof(int32_t) * (size_t)(ne > 0 ? ne : 1));
    if (!dsorted || !uniq) {
      free(dsorted);
      free(uniq);
      goto fail;
    }
    for (int64_t i = 0; i < nd; ++i) {
      dsorted[i].id = nodes[i];
      dsorted[i].pos = (int32_t)i;
    }
    qsort(dsorted, (size_t)nd, sizeof(orc_idpos), orc_cmp_idpos);
    memcpy(uniq, nbr, sizeof(int32_t) * (size_t)ne);
    qsort(uniq, (size_t)ne, sizeof(int32_t), orc_cmp_i32);
    int64_t n_new = 0;
    for (int64_t e = 0; e < ne; ++e) {
      if (e > 0 && uniq[e] == uniq[e - 1]) continue;
      if (orc_find_idpos(dsorted, nd, uniq[e]) >= 0) continue;
      uniq[n_new++] = uniq[e];
    }

    /* src_h = dst_h ++ new_h. */
    int32_t* grown =
        (int32_t*)realloc(nodes, sizeof(int32_t) * (size_t)(nd + n_new > 0 ? nd + n_new : 1));
    if (!grown) {
      free(dsorted);
      free(uniq);
      goto fail;
    }
    nodes = grown;
    memcpy(nodes + nd, uniq, sizeof(int32_t) * (size_t)n_new);
    n_nodes = nd + n_new;
    out->num_src[h] = n_nodes;

    /* Relabel: col[e] = index of nbr[e] in src_h. */
    int32_t* col = (int32_t*)malloc(sizeof(int32_t) * (size_t)(ne > 0 ? ne : 1));
    if (!col) {
      free(dsorted);
      free(uniq);
      goto fail;
    }
    out->col[h] = col;
    for (int64_t e = 0; e < ne; ++e) {
      int64_t d = orc_find_idpos(dsorted, nd, nbr[e]);
      if (d >= 0) {
        col[e] = dsorted[d].pos;
      } else {
        int64_t r = orc_find_i32(uniq, n_new, nbr[e]);
        col[e] = (int32_t)(nd + r);
      }
    }
    free(dsorted);
    free(uniq);

    /* Algorithm 1 read literally: the next frontier is N_out, the distinct
     * ids sampled at this hop, ascending (the last hop keeps src). */
    if (frontier_mode == ORC_FRONTIER_SAMPLED && h + 1 < K) {
      int32_t* sorted = (int32_t*)malloc(sizeof(int32_t) * (size_t)(ne > 0 ? ne : 1));
      if (!sorted) goto fail;
      memcpy(sorted, nbr, sizeof(int32_t) * (size_t)ne);
      qsort(sorted, (size_t)ne, sizeof(int32_t), orc_cmp_i32);
      int64_t n_out = 0; /* N_out is a subset of src_h, so it fits in nodes */
      for (int64_t e = 0; e < ne; ++e)
        if (e == 0 || sorted[e] != sorted[e - 1]) nodes[n_out++] = sorted[e];
      free(sorted);
      n_nodes = n_out;
    }
  }

  out->nodes = nodes;
  out->num_nodes = n_nodes;
  nodes = NULL;

  /* Gather: one feature row per node of src_K, copied byte for byte. */
  if (do_gather && g->features && g->row_bytes > 0) {
    size_t rb = (size_t)g->row_bytes;
    out->feats = (uint8_t*)malloc(rb * (size_t)(out->num_nodes > 0 ? out->num_nodes : 1));
    if (!out->feats) goto fail;
    for (int64_t r = 0; r < out->num_nodes; ++r)
      memcpy(out->feats + (size_t)r * rb, g->features + (size_t)out->nodes[r] * rb, rb);
  }
  return ORC_OK;

fail:
  free(nodes);
  orc_free_minibatch(out);
  return rc;
}

/* ---------------------------------------------------------------------
 * Blocks touched by a hyperbatch: the number of distinct adjacency blocks
 * that hold a node of some minibatch's frontier dst_h (the block-wise I/Os
 * of hop h, Sec. 3.3 and Fig. 7), and of distinct feature blocks holding a
 * node of some src_K (the gathering I/Os).
 * ------------------------------------------------------------------- */
int orc_hyperbatch_stats(const orc_graph* g, const orc_minibatch* mbs,
                         int32_t H, int64_t adj_block_bytes,
                         int64_t feat_rows_per_block, int64_t* out) {
  if (orc_check_graph(g) != ORC_OK || !mbs || H < 1 || !out ||
      feat_rows_per_block < 1)
    return ORC_EINVAL;
  const int32_t K = mbs[0].K;
  for (int32_t j = 1; j < H; ++j)
    if (mbs[j].K != K) return ORC_EINVAL;
  int32_t* node_block =
      (int32_t*)malloc(sizeof(int32_t) * (size_t)(g->num_nodes > 0 ? g->num_nodes : 1));
  if (!node_block) return ORC_ENOMEM;
  int64_t nb = 0;
  int rc = orc_build_adj_blocks(g, adj_block_bytes, node_block, &nb);
  if (rc != ORC_OK) {
    free(node_block);
    return rc;
  }
  int64_t nfb = (g->num_nodes + feat_rows_per_block - 1) / feat_rows_per_block;
  int64_t nmark = nb > nfb ? nb : nfb;
  uint8_t* mark = (uint8_t*)malloc((size_t)(nmark > 0 ? nmark : 1));
  if (!mark) {
    free(node_block);
    return ORC_ENOMEM;
  }
  for (int32_t h = 0; h < K; ++h) {
    memset(mark, 0, (size_t)(nmark > 0 ? nmark : 1));
    int64_t count = 0;
    for (int32_t j = 0; j < H; ++j) {
      for (int64_t i = 0; i < mbs[j].num_dst[h]; ++i) {
        int32_t b = node_block[mbs[j].dst[h][i]];
        if (!mark[b]) {
          mark[b] = 1;
          ++count;
        }
      }
    }
    out[h] = count;
  }
  memset(mark, 0, (size_t)(nmark > 0 ? nmark : 1));
  int64_t count = 0;
  for (int32_t j = 0; j < H; ++j) {
    for (int64_t i = 0; i < mbs[j].num_nodes; ++i) {
      int64_t b = (int64_t)mbs[j].nodes[i] / feat_rows_per_block;
      if (!mark[b]) {
        mark[b] = 1;
        ++count;
      }
    }
  }
  out[K] = count;
  free(mark);
  free(node_block);
  return ORC_OK;
}
