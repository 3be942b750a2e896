/* A plain C99 client of liblacache.so: the C ABI used without Python.
 *
 * Builds a cache of N random unit keys (fp32, rounded to bf16 by the library) with random unit prefix embeddings
 * and token ids, then looks up 8 queries from host memory with lacache_lookup_host:
 *   queries 0-3  exact copies of entries (key, prefix, ids)      -> HIT on that entry
 *   queries 4-5  an entry's key with a fresh prefix and fresh ids -> REJECT (the lookahead check fails)
 *   queries 6-7  fresh random keys                                -> MISS_KEY
 * Random unit vectors in d = 64 have |cos| < 0.9 with overwhelming probability, so every copied key's only
 * candidate is its own entry. The same batch then goes twice through lacache_lookup_host_async, from and into
 * mapped pinned buffers (cudaHostAlloc), both calls in flight on one stream before it is synchronized; both must
 * give the same decisions. Exits 0 and prints "ok" when every decision is as listed. */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "lacache.h"

enum { D = 64, K = 4, N = 4096, B = 8, TOP_C = 4 };

static uint64_t rng = 0x9E3779B97F4A7C15ull;
static double uniform(void) { /* xorshift64*, (0, 1) */
  rng ^= rng >> 12;
  rng ^= rng << 25;
  rng ^= rng >> 27;
  return ((rng * 0x2545F4914F6CDD1Dull) >> 11) * (1.0 / 9007199254740992.0) + 1e-300;
}
static void unit_vector(float* v) {
  double s = 0;
  for (int i = 0; i < D; i += 2) { /* Box-Muller */
    const double r = sqrt(-2.0 * log(uniform())), t = 6.283185307179586 * uniform();
    v[i] = (float)(r * cos(t));
    v[i + 1] = (float)(r * sin(t));
  }
  for (int i = 0; i < D; ++i) s += (double)v[i] * v[i];
  for (int i = 0; i < D; ++i) v[i] = (float)(v[i] / sqrt(s));
}
static uint16_t bf16(float f) { /* round to nearest even, as the library rounds fp32 inserts */
  uint32_t u;
  memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

#define CHECK(call)                                                              \
  do {                                                                           \
    lacache_status s_ = (call);                                                  \
    if (s_ != LACACHE_OK) {                                                      \
      fprintf(stderr, "%s: %s\n", #call, lacache_status_string(s_));             \
      return 1;                                                                  \
    }                                                                            \
  } while (0)

int main(void) {
  static float key[N * D], pre[N * D];
  static int32_t ids[N * K];
  for (int j = 0; j < N; ++j) {
    unit_vector(key + j * D);
    unit_vector(pre + j * D);
    for (int t = 0; t < K; ++t) ids[j * K + t] = (int32_t)(uniform() * 32000);
  }
  void *key_dev = NULL, *pre_dev = NULL, *ids_dev = NULL;
  if (cudaMalloc(&key_dev, sizeof key) != cudaSuccess || cudaMalloc(&pre_dev, sizeof pre) != cudaSuccess ||
      cudaMalloc(&ids_dev, sizeof ids) != cudaSuccess)
    return 1;
  cudaMemcpy(key_dev, key, sizeof key, cudaMemcpyHostToDevice);
  cudaMemcpy(pre_dev, pre, sizeof pre, cudaMemcpyHostToDevice);
  cudaMemcpy(ids_dev, ids, sizeof ids, cudaMemcpyHostToDevice);

  lacache_config cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.d = D;
  cfg.k = K;
  cfg.capacity = N;
  cfg.tau_c = 0.9f;
  cfg.tau_a = 0.8f;
  cfg.top_c = TOP_C;
  cfg.check_mode = LACACHE_CHECK_EMB;
  cfg.max_batch = B;
  cfg.device = 0;
  cfg.stage1 = LACACHE_STAGE1_AUTO;
  lacache_t* h = NULL;
  CHECK(lacache_create(&cfg, &h));
  int64_t first = -1, size = 0;
  CHECK(lacache_insert(h, N, key_dev, pre_dev, (const int32_t*)ids_dev, LACACHE_F32, &first, NULL));
  CHECK(lacache_sync(h));
  CHECK(lacache_size(h, &size));
  if (first != 0 || size != N) return 1;

  const int target[B] = {17, 1000, 2048, 4095, 321, 3210, -1, -1};
  const uint8_t want[B] = {LACACHE_HIT, LACACHE_HIT, LACACHE_HIT, LACACHE_HIT,
                           LACACHE_REJECT, LACACHE_REJECT, LACACHE_MISS_KEY, LACACHE_MISS_KEY};
  static uint16_t q_emb[B * D], q_pre[B * D];
  static int32_t q_ids[B * K];
  float tmp[D];
  for (int b = 0; b < B; ++b) {
    const int j = target[b];
    if (j >= 0) {
      for (int i = 0; i < D; ++i) q_emb[b * D + i] = bf16(key[j * D + i]);
    } else {
      unit_vector(tmp);
      for (int i = 0; i < D; ++i) q_emb[b * D + i] = bf16(tmp[i]);
    }
    if (j >= 0 && want[b] == LACACHE_HIT) {
      for (int i = 0; i < D; ++i) q_pre[b * D + i] = bf16(pre[j * D + i]);
      for (int t = 0; t < K; ++t) q_ids[b * K + t] = ids[j * K + t];
    } else {
      unit_vector(tmp);
      for (int i = 0; i < D; ++i) q_pre[b * D + i] = bf16(tmp[i]);
      for (int t = 0; t < K; ++t) q_ids[b * K + t] = (int32_t)(uniform() * 32000);
    }
  }
  int32_t entry_id[B], token_matches[B], n_cand[B];
  uint8_t status[B];
  float key_score[B], prefix_score[B];
  lacache_result out;
  memset(&out, 0, sizeof out);
  out.entry_id = entry_id;
  out.status = status;
  out.key_score = key_score;
  out.prefix_score = prefix_score;
  out.token_matches = token_matches;
  out.n_cand = n_cand;
  CHECK(lacache_lookup_host(h, B, q_emb, q_pre, q_ids, &out, NULL));
  CHECK(lacache_sync(h));
  int bad = 0;
  for (int b = 0; b < B; ++b) {
    const int want_id = want[b] == LACACHE_HIT ? target[b] : -1;
    const int want_n = target[b] >= 0 ? 1 : 0;
    if (status[b] != want[b] || entry_id[b] != want_id || n_cand[b] != want_n) {
      fprintf(stderr, "query %d: status %d entry %d n_cand %d key %.4f prefix %.4f\n", b, status[b], entry_id[b],
              n_cand[b], key_score[b], prefix_score[b]);
      bad = 1;
    }
  }

  /* the pipelined form: inputs and outputs in mapped pinned memory, two lookups in flight */
  struct Pinned {
    uint16_t emb[B * D], pre[B * D];
    int32_t ids[B * K];
    int32_t entry_id[2][B], token_matches[2][B], n_cand[2][B];
    float key_score[2][B], prefix_score[2][B];
    uint8_t status[2][B];
  }* pin = NULL;
  if (cudaHostAlloc((void**)&pin, sizeof *pin, cudaHostAllocMapped) != cudaSuccess) return 1;
  memcpy(pin->emb, q_emb, sizeof q_emb);
  memcpy(pin->pre, q_pre, sizeof q_pre);
  memcpy(pin->ids, q_ids, sizeof q_ids);
  cudaStream_t stream;
  if (cudaStreamCreate(&stream) != cudaSuccess) return 1;
  for (int r = 0; r < 2; ++r) {
    lacache_result o;
    memset(&o, 0, sizeof o);
    o.entry_id = pin->entry_id[r];
    o.status = pin->status[r];
    o.key_score = pin->key_score[r];
    o.prefix_score = pin->prefix_score[r];
    o.token_matches = pin->token_matches[r];
    o.n_cand = pin->n_cand[r];
    CHECK(lacache_lookup_host_async(h, B, pin->emb, pin->pre, pin->ids, &o, stream));
  }
  if (cudaStreamSynchronize(stream) != cudaSuccess) return 1;
  CHECK(lacache_sync(h));
  for (int r = 0; r < 2; ++r)
    for (int b = 0; b < B; ++b)
      if (pin->status[r][b] != status[b] || pin->entry_id[r][b] != entry_id[b] || pin->n_cand[r][b] != n_cand[b]) {
        fprintf(stderr, "async call %d, query %d: status %d entry %d\n", r, b, pin->status[r][b],
                pin->entry_id[r][b]);
        bad = 1;
      }
  cudaStreamDestroy(stream);
  cudaFreeHost(pin);

  CHECK(lacache_destroy(h));
  cudaFree(key_dev);
  cudaFree(pre_dev);
  cudaFree(ids_dev);
  if (bad) return 1;
  printf("ok\n");
  return 0;
}
