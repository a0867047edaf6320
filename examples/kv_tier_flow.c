/*
 * kv_tier_flow.c -- the shared-tier flow of two replicas from plain C: replica
 * A stores a prefix into the host tier under its chunk keys and commits them
 * on its stream; replica B finds the prefix, waits until it is readable,
 * acquires the entries on its own stream (which then waits for A's commits),
 * restores them into other pages and releases them.  Each replica has its own
 * context and stream; every byte restored is compared with its source.
 *
 * Build (with libkvxfer.so built in tree):
 *   gcc -O2 -I include examples/kv_tier_flow.c -o kv_tier_flow \
 *       -L paper_2609_15021_gb300/_lib -lkvxfer -L /usr/local/cuda/lib64 -lcudart \
 *       -Wl,-rpath,$PWD/paper_2609_15021_gb300/_lib -Wl,-rpath,/usr/local/cuda/lib64
 * Run: ./kv_tier_flow   (prints "tier flow ok" and exits 0 on success)
 */
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "kvxfer.h"

#define CHECK(x)                                                                              \
  do {                                                                                        \
    kvx_status s_ = (x);                                                                      \
    if (s_ != KVX_OK) {                                                                       \
      fprintf(stderr, "%s: %s (%s)\n", #x, kv_status_string(s_), kv_last_error_message()); \
      return 1;                                                                               \
    }                                                                                         \
  } while (0)

enum { L = 2, N = 32, B = 16, H = 2, D = 64, E = 2, C = 64, USED = 20, MAXC = 8 };

int main(void) {
  const int64_t page = 2LL * H * B * D * E, layer_bytes = N * page, tokens = USED * B - 3;
  void* src[L];
  void* dst[L];
  uint8_t* h_src = malloc(layer_bytes);
  uint8_t* h_dst = malloc(layer_bytes);
  for (int l = 0; l < L; ++l) {
    if (cudaMalloc(&src[l], layer_bytes) != cudaSuccess || cudaMalloc(&dst[l], layer_bytes) != cudaSuccess) return 1;
    for (int64_t i = 0; i < layer_bytes; ++i) h_src[i] = (uint8_t)(i * 37 + l * 11 + (i >> 11));
    cudaMemcpy(src[l], h_src, layer_bytes, cudaMemcpyHostToDevice);
    cudaMemset(dst[l], 0xA5, layer_bytes);
  }
  int32_t ta[USED], tb[USED];
  for (int i = 0; i < USED; ++i) {
    ta[i] = (i * 7 + 2) % N;   /* replica A's pages */
    tb[i] = (i * 13 + 5) % N;  /* replica B's freshly listed pages */
  }
  int32_t *d_ta, *d_tb;
  cudaMalloc((void**)&d_ta, sizeof(ta));
  cudaMalloc((void**)&d_tb, sizeof(tb));
  cudaMemcpy(d_ta, ta, sizeof(ta), cudaMemcpyHostToDevice);
  cudaMemcpy(d_tb, tb, sizeof(tb), cudaMemcpyHostToDevice);
  kvx_pool pa = {L, src, N, B, H, D, E, KVX_LAYOUT_HND, 1};
  kvx_pool pb = {L, dst, N, B, H, D, E, KVX_LAYOUT_HND, 1};
  kvx_chunk_layout lay;
  CHECK(kv_chunk_layout(&pa, C, C, &lay));
  const int n_chunks = (int)((tokens + C - 1) / C);

  /* the prefix's chunk keys: every chunk's key depends on all tokens before it */
  int32_t token_ids[USED * B];
  for (int t = 0; t < USED * B; ++t) token_ids[t] = (t * 7919) % 150001;
  uint64_t keys[MAXC];
  CHECK(kv_chunk_keys(token_ids, tokens, C, 42, keys, n_chunks));

  kvx_tier* tier = NULL;
  CHECK(kv_tier_create(lay.chunk_bytes, 2 * n_chunks, &tier));
  kvx_ctx *ctx_a = NULL, *ctx_b = NULL;
  CHECK(kv_ctx_create(0, NULL, &ctx_a));
  CHECK(kv_ctx_create(0, NULL, &ctx_b));
  cudaStream_t sa, sb;
  cudaStreamCreateWithFlags(&sa, cudaStreamNonBlocking);
  cudaStreamCreateWithFlags(&sb, cudaStreamNonBlocking);

  /* replica A: reserve a slot per key, store into the slots, commit on its stream */
  void* slots[MAXC];
  int64_t reserved = 0;
  CHECK(kv_tier_reserve_many(tier, keys, n_chunks, slots, &reserved));
  CHECK(kv_store(ctx_a, &pa, d_ta, USED, 0, tokens, C, slots, n_chunks, (kvx_stream_t)sa));
  CHECK(kv_tier_commit_many(tier, keys, n_chunks, (kvx_stream_t)sa));

  /* replica B: the cached prefix, a bounded wait until it is readable, then
     acquire (B's stream waits for A's commits), restore, release */
  int64_t hits = 0;
  CHECK(kv_tier_prefix_hits(tier, keys, n_chunks, &hits));
  CHECK(kv_tier_wait(tier, keys, hits, 10LL * 1000 * 1000 * 1000, NULL));
  void* found[MAXC];
  CHECK(kv_tier_acquire_many(tier, keys, hits, (kvx_stream_t)sb, found));
  CHECK(kv_load(ctx_b, &pb, d_tb, USED, 0, tokens, C, (const void* const*)found, hits, (kvx_stream_t)sb));
  CHECK(kv_tier_release_many(tier, keys, hits, (kvx_stream_t)sb));
  cudaStreamSynchronize(sb);
  cudaStreamSynchronize(sa);
  int64_t bad_a = 0, bad_b = 0;
  CHECK(kv_get_device_error(ctx_a, &bad_a));
  CHECK(kv_get_device_error(ctx_b, &bad_b));
  CHECK(kv_tier_poll(tier));
  kvx_tier_stats st;
  CHECK(kv_tier_stats(tier, &st));

  int errors = 0;
  for (int l = 0; l < L; ++l) {
    cudaMemcpy(h_src, src[l], layer_bytes, cudaMemcpyDeviceToHost);
    cudaMemcpy(h_dst, dst[l], layer_bytes, cudaMemcpyDeviceToHost);
    for (int64_t t = 0; t < tokens; ++t)
      for (int kv = 0; kv < 2; ++kv)
        for (int h = 0; h < H; ++h) {
          const int64_t row = D * E, s = t % B;
          const int64_t a = ta[t / B] * page + ((kv * H + h) * B + s) * row;
          const int64_t b = tb[t / B] * page + ((kv * H + h) * B + s) * row;
          errors += memcmp(h_src + a, h_dst + b, row) != 0;
        }
  }
  kv_ctx_destroy(ctx_a);
  kv_ctx_destroy(ctx_b);
  kv_tier_destroy(tier);
  if (errors || bad_a != -1 || bad_b != -1 || hits != n_chunks || reserved != n_chunks || st.pinned != 0) {
    fprintf(stderr, "tier flow failed: %d mismatches, hits %lld of %d, pinned %lld\n", errors, (long long)hits,
            n_chunks, (long long)st.pinned);
    return 1;
  }
  printf("tier flow ok: %d chunks stored by replica A, found, awaited, restored by replica B (%lld hits)\n",
         n_chunks, (long long)st.hits);
  return 0;
}
