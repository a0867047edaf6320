/*
 * kv_roundtrip.c -- the C ABI used from plain C: store a paged KV range into
 * pinned host chunks and restore it into other pages, then compare bytes.
 *
 * Build (with libkvxfer.so built in tree):
 *   gcc -O2 -I include examples/kv_roundtrip.c -o kv_roundtrip \
 *       -L paper_2609_15021_gb300/_lib -lkvxfer -L /usr/local/cuda/lib64 -lcudart \
 *       -Wl,-rpath,$PWD/paper_2609_15021_gb300/_lib -Wl,-rpath,/usr/local/cuda/lib64
 * Run: ./kv_roundtrip   (prints "roundtrip ok" and exits 0 on success)
 */
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "kvxfer.h"

#define CHECK(x)                                                          \
  do {                                                                    \
    kvx_status s_ = (x);                                                  \
    if (s_ != KVX_OK) {                                                   \
      fprintf(stderr, "%s: %s (%s)\n", #x, kv_status_string(s_), kv_last_error_message()); \
      return 1;                                                           \
    }                                                                     \
  } while (0)

int main(void) {
  enum { L = 2, N = 16, B = 16, H = 2, D = 64, E = 2, C = 64, USED = 10 };
  const int64_t page = 2LL * H * B * D * E, layer_bytes = N * page, tokens = USED * B - 5;
  void* src[L];
  void* dst[L];
  uint8_t* host_src = malloc(layer_bytes);
  uint8_t* host_dst = malloc(layer_bytes);
  for (int l = 0; l < L; ++l) {
    if (cudaMalloc(&src[l], layer_bytes) != cudaSuccess || cudaMalloc(&dst[l], layer_bytes) != cudaSuccess) return 1;
    for (int64_t i = 0; i < layer_bytes; ++i) host_src[i] = (uint8_t)(i * 131 + l * 7 + (i >> 9));
    cudaMemcpy(src[l], host_src, layer_bytes, cudaMemcpyHostToDevice);
    cudaMemset(dst[l], 0xA5, layer_bytes);
  }
  int32_t ta[USED], tb[USED];
  for (int i = 0; i < USED; ++i) {
    ta[i] = (i * 5 + 3) % N;  /* two different permutations of pages */
    tb[i] = (i * 7 + 1) % N;
  }
  int32_t *d_ta, *d_tb;
  cudaMalloc((void**)&d_ta, sizeof(ta));
  cudaMalloc((void**)&d_tb, sizeof(tb));
  cudaMemcpy(d_ta, ta, sizeof(ta), cudaMemcpyHostToDevice);
  cudaMemcpy(d_tb, tb, sizeof(tb), cudaMemcpyHostToDevice);

  kvx_pool ps = {L, src, N, B, H, D, E, KVX_LAYOUT_HND, 1};
  kvx_pool pd = {L, dst, N, B, H, D, E, KVX_LAYOUT_HND, 1};
  kvx_chunk_layout lay;
  CHECK(kv_chunk_layout(&ps, C, C, &lay));
  const int n_chunks = (int)((tokens + C - 1) / C);
  void* pool = NULL;
  CHECK(kv_host_alloc(n_chunks * lay.chunk_bytes, &pool));
  void* chunks[8];
  for (int i = 0; i < n_chunks; ++i) chunks[i] = (uint8_t*)pool + i * lay.chunk_bytes;

  kvx_ctx* ctx = NULL;
  CHECK(kv_ctx_create(0, NULL, &ctx));
  cudaStream_t s;
  cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
  CHECK(kv_store(ctx, &ps, d_ta, USED, 0, tokens, C, chunks, n_chunks, (kvx_stream_t)s));
  CHECK(kv_load(ctx, &pd, d_tb, USED, 0, tokens, C, (const void* const*)chunks, n_chunks, (kvx_stream_t)s));
  cudaStreamSynchronize(s);
  int64_t bad = 0;
  CHECK(kv_get_device_error(ctx, &bad));

  /* every restored token row equals its source row; every other byte is untouched */
  int errors = 0;
  for (int l = 0; l < L; ++l) {
    cudaMemcpy(host_src, src[l], layer_bytes, cudaMemcpyDeviceToHost);
    cudaMemcpy(host_dst, dst[l], layer_bytes, cudaMemcpyDeviceToHost);
    uint8_t* touched = calloc(layer_bytes, 1);
    for (int64_t t = 0; t < tokens; ++t)
      for (int kv = 0; kv < 2; ++kv)
        for (int h = 0; h < H; ++h) {
          const int64_t row = D * E, s_ = t % B;
          const int64_t a = ta[t / B] * page + ((kv * H + h) * B + s_) * row;
          const int64_t b = tb[t / B] * page + ((kv * H + h) * B + s_) * row;
          errors += memcmp(host_src + a, host_dst + b, row) != 0;
          memset(touched + b, 1, row);
        }
    for (int64_t i = 0; i < layer_bytes; ++i) errors += !touched[i] && host_dst[i] != 0xA5;
    free(touched);
  }
  kv_ctx_destroy(ctx);
  kv_host_free(pool);
  if (errors || bad != -1) {
    fprintf(stderr, "roundtrip failed: %d mismatches, bad block %lld\n", errors, (long long)bad);
    return 1;
  }
  printf("roundtrip ok: %lld tokens in %d chunks of %lld bytes\n", (long long)tokens, n_chunks,
         (long long)lay.chunk_bytes);
  return 0;
}
