/*
 * kv_oracle.c -- CPU oracle for the paged-KV <-> packed-host-chunk byte move.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or
 * call this file; only the test suite, the smoke check and the CPU-baseline
 * leg of the benchmark do.  It shares no code, header or constant with the
 * CUDA library: everything below is written out again from the definition.
 *
 * What it computes (paper, Sec. 2.1 Table 1 and Sec. 3.1: a paged GPU KV cache
 * whose logical blocks are pages of the pool, stored to a shared host tier in
 * fixed-token chunks; Sec. 3.2: the store is a gather of those pages into the
 * chunk and the load is the scatter back into freshly allocated pages):
 *
 *   layer l of the pool is an array of num_blocks pages; a page holds K (kv=0)
 *   then V (kv=1), each as
 *       HND: [num_heads][block_tokens][row]      (the paper's layout, Table 1)
 *       NHD: [block_tokens][num_heads][row]
 *   where a row is head_dim * elem_bytes bytes (one head vector of one token).
 *
 *   The block table names logical blocks of P = pages_per_block packed
 *   pages (Sec. 3.1: a 1,568-token logical block spans 49 pages of 32
 *   tokens); logical block b holds pages b*P .. b*P + P-1 of the pool.
 *   Token t lies in kernel page k = t / B at slot s = t % B; its page is
 *       p = table[k / P] * P + k % P          (P = 1: p = table[t / B]).
 *
 *   chunk c covers tokens [c*C, min((c+1)*C, t_end)); it is laid out
 *       [layer][kv][u][head][row],  u = t - c*C,  T_c tokens per chunk,
 *   densely, so a partial last chunk is shorter, not padded.
 *
 *   store: chunk_c[l][kv][u][h] = pool_l[p][kv][h][s]  (HND)
 *                                 pool_l[p][kv][s][h]  (NHD)
 *   load : the same equation read right to left, into a different table.
 *
 * Bytes are moved with memcpy, one row at a time.  Bytes of a chunk past its
 * L*2*T_c*H*row valid bytes, and pool bytes of token slots outside
 * [t_begin, t_end), are never written.  A table entry outside
 * [0, num_blocks) names no page: a store writes zero bytes for its tokens,
 * a load writes nothing for them, and the lowest offending logical block
 * index is reported.  (The paper does not define this case.)
 *
 * Recurrent-state snapshots (Sec. 2.2: a recurrent page is handled as opaque
 * addressable bytes) are a plain byte copy of one slot per layer.
 *
 * Work may be split over threads by chunk; chunks touch disjoint bytes.
 */
#include <stdint.h>
#include <string.h>
#include <pthread.h>

/* status values (the oracle's own; the test suite maps them) */
#define OR_OK 0
#define OR_EINVAL (-1)
#define OR_EALIGN (-2)
#define OR_ERANGE (-3)

#define OR_HND 0
#define OR_NHD 1

typedef struct {
  int32_t num_layers;
  int64_t num_blocks;
  int32_t block_tokens; /* B */
  int32_t num_heads;    /* H */
  int32_t head_dim;     /* D */
  int32_t elem_bytes;   /* e */
  int32_t layout;       /* OR_HND or OR_NHD */
  int32_t pages_per_block; /* P: pages per logical block of the table (0 means 1) */
} or_pool;

static int64_t ppb_of(const or_pool* P) { return P->pages_per_block > 1 ? P->pages_per_block : 1; }

static int64_t row_bytes(const or_pool* P) { return (int64_t)P->head_dim * P->elem_bytes; }

/* byte offset, inside one layer of the pool, of the row (page p, kv, head h, slot s) */
static int64_t page_row(const or_pool* P, int64_t p, int64_t kv, int64_t h, int64_t s) {
  int64_t H = P->num_heads, B = P->block_tokens;
  if (P->layout == OR_HND)
    return (((p * 2 + kv) * H + h) * B + s) * row_bytes(P);
  return (((p * 2 + kv) * B + s) * H + h) * row_bytes(P);
}

/* byte offset, inside one chunk of T_c tokens, of the row (layer l, kv, token u, head h) */
static int64_t chunk_row(const or_pool* P, int64_t T_c, int64_t l, int64_t kv, int64_t u, int64_t h) {
  int64_t H = P->num_heads;
  return (((l * 2 + kv) * T_c + u) * H + h) * row_bytes(P);
}

/* the argument rules both directions share */
static int check_args(const or_pool* P, int64_t table_len, int64_t t_begin, int64_t t_end,
                      int32_t C, int64_t n_chunks) {
  if (!P || P->num_layers < 1 || P->num_blocks < 1 || P->block_tokens < 1 || P->num_heads < 1 ||
      P->head_dim < 1 || P->elem_bytes < 1 || (P->layout != OR_HND && P->layout != OR_NHD) ||
      C < 1 || table_len < 0 || n_chunks < 0)
    return OR_EINVAL;
  if (P->pages_per_block < 0) return OR_EINVAL;
  if (P->num_blocks % ppb_of(P) != 0) return OR_EALIGN;
  if (t_begin < 0 || t_end < t_begin) return OR_ERANGE;
  if (C % P->block_tokens != 0) return OR_EALIGN;
  if (t_begin % C != 0) return OR_EALIGN;
  if (t_end > table_len * ppb_of(P) * (int64_t)P->block_tokens) return OR_ERANGE;
  {
    int64_t first = t_begin / C;
    int64_t last = (t_end + C - 1) / C; /* one past the last chunk */
    if (t_end > t_begin && last - first > n_chunks) return OR_ERANGE;
  }
  return OR_OK;
}

typedef struct {
  const or_pool* P;
  uint8_t* const* layers;
  const int32_t* table;
  int64_t t_begin, t_end;
  int32_t C;
  uint8_t* const* chunks;
  int to_chunk;        /* 1 = store (pool -> chunk), 0 = load (chunk -> pool) */
  int64_t c_lo, c_hi;  /* chunk indices, relative to t_begin / C */
  int64_t bad;         /* lowest logical block with an out-of-range entry, or -1 */
} or_job;

static void* run_job(void* arg) {
  or_job* J = (or_job*)arg;
  const or_pool* P = J->P;
  int64_t B = P->block_tokens, C = J->C, row = row_bytes(P), ppb = ppb_of(P);
  int64_t c0 = J->t_begin / C;
  for (int64_t i = J->c_lo; i < J->c_hi; ++i) {
    int64_t c = c0 + i;
    int64_t first = c * C;
    int64_t T_c = (J->t_end - first < C) ? (J->t_end - first) : C;
    uint8_t* chunk = J->chunks[i];
    for (int64_t l = 0; l < P->num_layers; ++l)
      for (int64_t kv = 0; kv < 2; ++kv)
        for (int64_t u = 0; u < T_c; ++u) {
          int64_t t = first + u;
          int64_t kpage = t / B;            /* kernel page of the token */
          int64_t blk = kpage / ppb;        /* logical block in the table */
          int64_t s = t % B;
          int64_t entry = J->table[blk];
          int64_t p = entry * ppb + kpage % ppb;
          if (entry < 0 || entry >= P->num_blocks / ppb) {
            if (J->bad < 0 || blk < J->bad) J->bad = blk;
            if (J->to_chunk) /* the token's rows of this (layer, kv) read as zeros */
              memset(chunk + chunk_row(P, T_c, l, kv, u, 0), 0, (size_t)(P->num_heads * row));
            continue;
          }
          for (int64_t h = 0; h < P->num_heads; ++h) {
            uint8_t* c_ptr = chunk + chunk_row(P, T_c, l, kv, u, h);
            uint8_t* p_ptr = J->layers[l] + page_row(P, p, kv, h, s);
            if (J->to_chunk)
              memcpy(c_ptr, p_ptr, (size_t)row);
            else
              memcpy(p_ptr, c_ptr, (size_t)row);
          }
        }
  }
  return 0;
}

static int run(const or_pool* P, uint8_t* const* layers, const int32_t* table, int64_t table_len,
               int64_t t_begin, int64_t t_end, int32_t C, uint8_t* const* chunks, int64_t n_chunks,
               int to_chunk, int n_threads, int64_t* bad_block) {
  int rc = check_args(P, table_len, t_begin, t_end, C, n_chunks);
  if (bad_block) *bad_block = -1;
  if (rc != OR_OK) return rc;
  if (t_end == t_begin) return OR_OK;
  int64_t n = (t_end + C - 1) / C - t_begin / C;
  if (n_threads < 1) n_threads = 1;
  if (n_threads > 256) n_threads = 256;
  if (n_threads > n) n_threads = (int)n;
  or_job jobs[256];
  pthread_t tid[256];
  for (int k = 0; k < n_threads; ++k) {
    or_job J = {P, layers, table, t_begin, t_end, C, chunks, to_chunk,
                n * k / n_threads, n * (k + 1) / n_threads, -1};
    jobs[k] = J;
  }
  int started = 0;
  for (int k = 1; k < n_threads; ++k) {
    if (pthread_create(&tid[k], 0, run_job, &jobs[k]) != 0) break;
    started = k;
  }
  run_job(&jobs[0]);
  for (int k = 1; k <= started; ++k) pthread_join(tid[k], 0);
  for (int k = started + 1; k < n_threads; ++k) run_job(&jobs[k]); /* threads that failed to start */
  int64_t bad = -1;
  for (int k = 0; k < n_threads; ++k)
    if (jobs[k].bad >= 0 && (bad < 0 || jobs[k].bad < bad)) bad = jobs[k].bad;
  if (bad_block) *bad_block = bad;
  return OR_OK;
}

/* store: gather the pages of [t_begin, t_end) into chunks[0 .. n_chunks) */
int oracle_store(const or_pool* P, uint8_t* const* layers, const int32_t* table, int64_t table_len,
                 int64_t t_begin, int64_t t_end, int32_t C, uint8_t* const* chunks, int64_t n_chunks,
                 int n_threads, int64_t* bad_block) {
  return run(P, layers, table, table_len, t_begin, t_end, C, chunks, n_chunks, 1, n_threads, bad_block);
}

/* load: scatter chunks[0 .. n_chunks) into the pages of [t_begin, t_end) */
int oracle_load(const or_pool* P, uint8_t* const* layers, const int32_t* table, int64_t table_len,
                int64_t t_begin, int64_t t_end, int32_t C, uint8_t* const* chunks, int64_t n_chunks,
                int n_threads, int64_t* bad_block) {
  return run(P, layers, table, table_len, t_begin, t_end, C, chunks, n_chunks, 0, n_threads, bad_block);
}

/* bytes of one chunk holding T_c tokens */
int64_t oracle_chunk_bytes(const or_pool* P, int64_t T_c) {
  return (int64_t)P->num_layers * 2 * T_c * P->num_heads * row_bytes(P);
}

/*
 * Recurrent-state snapshot (Sec. 2.2): layer l holds num_slots slots of
 * slot_bytes opaque bytes each.  The host object is [layer][slot_bytes].
 * to_host = 1 copies slot `slot` of every layer out; 0 copies it back in.
 */
int oracle_state_copy(int32_t num_layers, uint8_t* const* layers, int64_t num_slots, int64_t slot_bytes,
                      int64_t slot, uint8_t* host_obj, int to_host) {
  if (num_layers < 1 || num_slots < 1 || slot_bytes < 1) return OR_EINVAL;
  if (slot < 0 || slot >= num_slots) return OR_ERANGE;
  for (int64_t l = 0; l < num_layers; ++l) {
    uint8_t* s = layers[l] + slot * slot_bytes;
    uint8_t* h = host_obj + l * slot_bytes;
    if (to_host)
      memcpy(h, s, (size_t)slot_bytes);
    else
      memcpy(s, h, (size_t)slot_bytes);
  }
  return OR_OK;
}
