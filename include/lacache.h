/*
 * lacache.h -- C ABI of the GB300 (sm_103a) LaCache lookup library, liblacache.so.
 *
 * LaCache ("LaCache: Robust Semantic Caching for LLM Serving") stores each cache entry as
 * <h(x), [h(f_k(x)), f(x)]> (section 3.2, "Cache Structure"): the key embedding of query x, the embedding of the
 * first k tokens of its response f_k(x), and the response. A query x is served from entry x' only if both checks
 * pass (Algorithm 1; section 4.1, "Metrics"):
 *     stage 1, key check:        sim(x, x')           >= tau_c
 *     stage 2, lookahead check:  sim(f_k(x), f_k(x')) >= tau_a
 * Otherwise x is decoded from scratch and its entry is appended to the cache (Algorithm 1, last two steps).
 *
 * This library is that lookup, batched, on one GPU. The response f(x) is the caller's: the library returns the
 * entry id, which stands for it. sim is the inner product of unit-norm embeddings (their cosine).
 *
 * Conventions for every call
 *  - Embeddings are bf16 (IEEE binary32 upper halves) in row-major [rows x d] layout. Token ids are int32 in
 *    row-major [rows x k] layout. All rows are dense (row stride d or k elements).
 *  - Pointers named *_dev are CUDA device pointers (cudaMalloc or equivalent) on the handle's device. Pointers
 *    named *_host are host pointers (page-locked memory is fastest). The caller owns every input and output
 *    buffer; the handle owns the device store and its scratch.
 *  - Device embedding pointers must be 16-byte aligned (TMA reads them). Host pointers may have any alignment.
 *  - `cuda_stream` is a cudaStream_t (NULL = the legacy default stream). Device calls are asynchronous on it;
 *    argument errors are reported synchronously and leave the cache unchanged.
 *  - Device-side faults of the library's own kernels (a bounded wait that ran out) do not abort the process:
 *    they set a status word that lacache_sync() reports as LACACHE_ERR_DEVICE_TIMEOUT.
 *  - A handle is not thread-safe. Lookups see every insert issued before them on the same stream.
 */
#ifndef LACACHE_H_
#define LACACHE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct lacache lacache_t; /* opaque */

typedef enum {
  LACACHE_OK = 0,
  LACACHE_ERR_INVALID_ARG = 1,    /* bad pointer, size, alignment or parameter */
  LACACHE_ERR_CAPACITY = 2,       /* an insert would exceed the capacity; nothing was inserted */
  LACACHE_ERR_OOM = 3,            /* device allocation failed at create */
  LACACHE_ERR_CUDA = 4,           /* a CUDA runtime call failed */
  LACACHE_ERR_DEVICE_TIMEOUT = 5, /* a kernel's bounded wait ran out (reported by lacache_sync) */
  LACACHE_ERR_UNSUPPORTED = 6,    /* valid but unsupported configuration (e.g. top_c > 32, d % 8 != 0) */
  LACACHE_ERR_IO = 7              /* a file could not be opened, read or written, or is not a saved cache */
} lacache_status;

/* How stage 2 decides that candidate x' passes the lookahead check (Algorithm 1; section 4.1). */
typedef enum {
  LACACHE_CHECK_EMB = 0,    /* sim(f_k(x), f_k(x')) >= tau_a, the form the paper evaluates */
  LACACHE_CHECK_TOKENS = 1, /* >= token_match_min of the k prefix token ids equal position by position;
                               token_match_min = k is Algorithm 1's h(f_k(x')) = h(f_k(x)) on ids */
  LACACHE_CHECK_BOTH = 2    /* both of the above */
} lacache_check_mode;

typedef enum { LACACHE_BF16 = 0, LACACHE_F32 = 1 } lacache_dtype;

/* Which stage-1 kernel lookups run. */
typedef enum {
  LACACHE_STAGE1_AUTO = 0,   /* the streaming scan when n x d x B <= 2^25 (few enough multiply-adds that its
                                latency is the shorter: at most 64 MiB of keys at one query) and for 1 or 2
                                queries at d = 1024 (where it matches the tensor-core scan from HBM); the
                                tensor-core scan otherwise, which holds the HBM roofline at every batch size */
  LACACHE_STAGE1_TENSOR = 1, /* tcgen05 tensor-core scan (TMA-fed, TMEM accumulators) */
  LACACHE_STAGE1_STREAM = 2, /* streaming CUDA-core scan: warp per key tile, 128-bit key loads, packed fp32 FMA */
  LACACHE_STAGE1_LSH = 3,    /* SimHash index, then the exact key check (requires lacache_enable_lsh) */
  LACACHE_STAGE1_TENSOR_PAIR = 4, /* reported by lacache_last_launch only, not a configuration value: the tensor
                                     scan on two-CTA clusters (one M=256 MMA per pair of SMs), chosen for batches
                                     of more than 128 queries */
  LACACHE_STAGE1_LSH_TENSOR = 5   /* reported by lacache_last_launch only: the SimHash form with the Hamming test on
                                     the tensor cores, chosen for batches of at least 48 queries at 256 bits
                                     and of at least 40 at 128 and 512 bits */
} lacache_stage1;

/* Ensemble of m lookahead checks (section 3.4, "Analysis"; Figure 6): every entry and query carries one k-token
 * prefix embedding per embedding model, concatenated in one prefix row of dims[0] + ... + dims[m-1] values, and a
 * candidate passes the lookahead check only if sim_i(f_k(x), f_k(x')) >= tau_a[i] for every model i. */
#define LACACHE_MAX_MODELS 8
typedef struct {
  int32_t m;                         /* number of lookahead checks, 1..LACACHE_MAX_MODELS */
  int32_t dims[LACACHE_MAX_MODELS];  /* each model's prefix embedding dimension (multiple of 8) */
  float tau_a[LACACHE_MAX_MODELS];   /* each model's lookahead threshold */
} lacache_ensemble;

/* Per-query status codes written to lacache_result.status. */
enum { LACACHE_MISS_KEY = 0, LACACHE_HIT = 1, LACACHE_REJECT = 2 };

typedef struct {
  int32_t d;               /* embedding dimension of keys and prefix embeddings; multiple of 8, <= 8192 */
  int32_t k;               /* lookahead window: token ids per entry, 1..256 */
  int64_t capacity;        /* maximum number of entries (device store is allocated once, at create) */
  float tau_c;             /* key threshold */
  float tau_a;             /* lookahead threshold */
  int32_t top_c;           /* candidates kept from stage 1 per query, 1..32 */
  int32_t token_match_min; /* LACACHE_CHECK_TOKENS/BOTH: positions that must match; <= 0 means k */
  int32_t check_mode;      /* lacache_check_mode */
  int32_t max_batch;       /* largest B passed to lookup; sizes the scratch and host-staging buffers */
  int32_t device;          /* CUDA device ordinal */
  int32_t stage1;          /* lacache_stage1 */
} lacache_config;

/* Per-query outputs of a lookup, each [B] (or [B x top_c] for the optional cand_* arrays). All device pointers
 * for lacache_lookup, host pointers for lacache_lookup_host. The cand_* arrays may be NULL (not written). */
typedef struct {
  int32_t* entry_id;          /* served entry j* on HIT, else -1 */
  uint8_t* status;            /* LACACHE_MISS_KEY / LACACHE_HIT / LACACHE_REJECT */
  float* key_score;           /* sim(x, x') of j* on HIT; otherwise the best key score over all entries
                                 (-inf for an empty cache) */
  float* prefix_score;        /* sim(f_k(x), f_k(x')) of j* on HIT, of the first candidate on REJECT; NaN on
                                 MISS_KEY */
  int32_t* token_matches;     /* equal token ids (positionwise) for the same candidate as prefix_score; -1 on
                                 MISS_KEY */
  int32_t* n_cand;            /* number of candidates |C_q| <= top_c */
  int32_t* cand_id;           /* optional [B x top_c]: C_q by (key score desc, id asc), -1 padded */
  float* cand_score;          /* optional [B x top_c]: their key scores, NaN padded */
  float* cand_prefix_score;   /* optional [B x top_c]: their lookahead scores, NaN padded */
  int32_t* cand_matches;      /* optional [B x top_c]: their token matches, -1 padded */
  float* prefix_scores;       /* optional [B x m]: every model's lookahead score for the candidate of prefix_score
                                 (prefix_score is model 0's); NaN on MISS_KEY */
  uint8_t* cand_pass;         /* optional [B x top_c]: 1 if the candidate passes the lookahead check under the
                                 handle's check mode (every model of an ensemble), 0 otherwise and as padding */
  float* cand_prefix_scores;  /* optional [B x top_c x m]: every model's lookahead score per candidate, NaN padded */
} lacache_result;

/* Create a cache on cfg->device with an empty store of cfg->capacity entries. Allocates the store
 * (capacity * (2d + 2 * prefix row + 4k) bytes), the stage-1 scratch (S * max_batch * (8 * top_c + 8) bytes for
 * S = 2 x SMs partial lists, or up to 4 x SMs while S * max_batch * top_c * 8 stays within 1 GiB) and host staging.
 * On success *out is a new handle; on failure *out is NULL and nothing stays allocated. */
lacache_status lacache_create(const lacache_config* cfg, lacache_t** out);

/* lacache_create for an ensemble of lookahead checks. cfg->tau_a is ignored; prefix rows everywhere (insert,
 * lookup, append, read_rows) are dims[0] + ... + dims[m-1] values long. lacache_create(cfg) is this call with
 * m = 1, dims = {cfg->d}, tau_a = {cfg->tau_a}. */
lacache_status lacache_create_ensemble(const lacache_config* cfg, const lacache_ensemble* ens, lacache_t** out);

/* Free the handle and everything it owns. Synchronizes the device first. NULL is accepted. */
lacache_status lacache_destroy(lacache_t* h);

/* Append n entries (Algorithm 1, "add <h(x), [h(f_k(x)), f(x)]> to cache"). key_dev is [n x d] and prefix_dev
 * [n x prefix row] in `dtype` (LACACHE_F32 rows are rounded to bf16, to nearest even, on the device); ids_dev is
 * [n x k] int32. All-or-nothing: if size + n > capacity, returns LACACHE_ERR_CAPACITY and inserts nothing. The new
 * entries get ids first_id .. first_id + n - 1 (first_id may be NULL). Asynchronous on cuda_stream. */
lacache_status lacache_insert(lacache_t* h, int64_t n, const void* key_dev, const void* prefix_dev,
                              const int32_t* ids_dev, int32_t dtype, int64_t* first_id, void* cuda_stream);

/* Batched two-stage lookup of B queries (1 <= B <= max_batch): q_emb_dev [B x d] bf16 key embeddings of the
 * queries, q_prefix_dev [B x prefix row] bf16 embeddings of their speculatively decoded k-token prefixes f_k(x),
 * q_ids_dev [B x k] int32 those token ids. Stage 1 keeps per query the top_c entries with key score >= tau_c by
 * (score desc, id asc); stage 2 checks them in that order and serves the first that passes. Writes every
 * non-NULL field of *out (device pointers). Asynchronous on cuda_stream; no host synchronization. Back-to-back
 * lookups on one stream overlap: a lookup's stage 1 scans while the previous lookup's stage 2 finishes, so the
 * query inputs of a lookup must not alias the output arrays of the lookup issued just before it on the stream
 * (any other work issued in between orders them as usual). The call may be captured into a CUDA graph (stream
 * capture). Replays then read the captured input and output pointers, and scan
 * the entries present at capture time: capture again after inserts or appends. */
lacache_status lacache_lookup(lacache_t* h, int32_t B, const void* q_emb_dev, const void* q_prefix_dev,
                              const int32_t* q_ids_dev, const lacache_result* out, void* cuda_stream);

/* lacache_lookup for host-resident queries and results (any host memory: pageable or pinned, any alignment).
 * The inputs reach the handle's device staging in one of two ways. An array in pinned memory that the device can
 * map is read by the device directly, one gather kernel covering all such arrays. Any other array is copied by
 * DMA. The same kernels then run. Their results go straight into the handle's mapped pinned staging, or through
 * one device-to-host copy where the device cannot map it. The call synchronizes cuda_stream, copies the results
 * into *out_host (host pointers) and returns. */
lacache_status lacache_lookup_host(lacache_t* h, int32_t B, const void* q_emb_host, const void* q_prefix_host,
                                   const int32_t* q_ids_host, const lacache_result* out_host, void* cuda_stream);

/* lacache_lookup_host without the synchronization, for pipelined serving: a caller may keep several lookups in
 * flight on one stream, each with its own output arrays. Every input array and every non-NULL field of *out_host
 * must lie in pinned host memory that the handle's device can map (cudaHostAlloc or cudaMallocHost, or
 * cudaHostRegister with mapping; with unified addressing all pinned memory is mapped), and each output field must
 * be aligned to its element size; otherwise the call returns LACACHE_ERR_INVALID_ARG and runs nothing. One kernel
 * gathers the inputs into the handle's device staging, the lookup's kernels follow, and they write the results
 * straight into the output arrays. The call returns once they are enqueued on cuda_stream. The output arrays hold
 * the results, and the input arrays may be reused, only after the stream has passed the call (an event recorded
 * after it, or cudaStreamSynchronize). Calls on one handle must all use one stream: the staging is the handle's. */
lacache_status lacache_lookup_host_async(lacache_t* h, int32_t B, const void* q_emb_host, const void* q_prefix_host,
                                         const int32_t* q_ids_host, const lacache_result* out_host,
                                         void* cuda_stream);

/* The cache update of the serve loop: append, in query order, every query of a looked-up batch whose status is
 * not LACACHE_HIT (a key miss or a lookahead rejection is decoded from scratch and added; Algorithm 1). The
 * inputs are those of the lookup (device pointers) and its status_dev output. The rows are gathered on the
 * device; the count is read back, so this call synchronizes cuda_stream. All-or-nothing on capacity. Writes the
 * first new id and the number appended (either pointer may be NULL). */
lacache_status lacache_append_misses(lacache_t* h, int32_t B, const void* q_emb_dev, const void* q_prefix_dev,
                                     const int32_t* q_ids_dev, const uint8_t* status_dev, int64_t* first_id,
                                     int64_t* n_appended, void* cuda_stream);

/* The SimHash index of Eq. 1 (section 2; Algorithm 1's "search semantic cache with key h(x)"). Every entry gets a
 * signature of `bits` bits (128, 256 or 512): bit i is set iff <r_i, key> >= 0 for the i-th row r_i of
 * hyperplanes_dev ([bits x d] bf16, copied into the handle; random normal rows give random-hyperplane LSH). With
 * cfg->stage1 == LACACHE_STAGE1_LSH a lookup applies the exact key check only to the entries whose signature
 * differs from the query's in at most `radius` bits; stage 2 is unchanged. Existing entries are signed now and
 * later inserts and appends are signed as they arrive. Batches of fewer than T queries (T = 48 at 256 bits, 40 at
 * 128 and 512) compare the packed signatures by population counts; larger ones run the Hamming test on the tensor
 * cores, over a copy of the signatures expanded to one byte per bit. Allocates (capacity + max_batch) * bits / 8
 * bytes for the signatures and, when max_batch >= T, capacity * bits bytes (whole 128-entry blocks) for the
 * expanded copy.
 * Asynchronous on cuda_stream; calling it again replaces the index. A lookup on a handle whose cfg->stage1 is
 * LACACHE_STAGE1_LSH returns LACACHE_ERR_INVALID_ARG, and runs nothing, until this call has been made. */
lacache_status lacache_enable_lsh(lacache_t* h, int32_t bits, int32_t radius, const void* hyperplanes_dev,
                                  void* cuda_stream);

/* Copy the SimHash signatures of entries [first, first + n) into sig_dev ([n x bits/32] uint32 words; bit i of
 * word w is hyperplane 32w + i). LACACHE_ERR_INVALID_ARG if the index is not enabled. Asynchronous. */
lacache_status lacache_read_signatures(const lacache_t* h, int64_t first, int64_t n, uint32_t* sig_dev,
                                       void* cuda_stream);

/* Copy entries [first, first + n) of the store into caller device buffers (key_dev [n x d], prefix_dev
 * [n x prefix row] bf16, ids_dev [n x k]); any of the three may be NULL. For checkpoints and checks. Asynchronous on
 * cuda_stream. */
lacache_status lacache_read_rows(const lacache_t* h, int64_t first, int64_t n, void* key_dev, void* prefix_dev,
                                 int32_t* ids_dev, void* cuda_stream);

/* Number of valid entries (as of the calls issued so far). */
lacache_status lacache_size(const lacache_t* h, int64_t* n);

/* Synchronize the handle's device and report any device-side status set by the library's kernels since the
 * previous lacache_sync (the status word is then cleared). */
lacache_status lacache_sync(lacache_t* h);

/* Persistence of a cache across processes. lacache_save writes the handle's configuration (lacache_config and the
 * lacache_ensemble of its lookahead checks) and its valid entries to `path`: an 8-byte magic "LACACHE1", a format
 * version, the two structs and the entry count, then the key rows [n x d] bf16, the prefix rows [n x prefix row]
 * bf16 and the token ids [n x k] int32, all little-endian. It synchronizes the handle's device first, so every
 * insert and append issued before the call is saved. A SimHash index is not saved: enable it again after loading.
 * lacache_load creates a new handle on `device` from such a file, with the saved configuration; capacity > 0
 * replaces the saved capacity (it must hold the saved entries, else LACACHE_ERR_CAPACITY). Entry ids are kept.
 * A file that cannot be read, or is not a saved cache, gives LACACHE_ERR_IO before any device is touched. */
lacache_status lacache_save(lacache_t* h, const char* path);
/* The handle's configuration and lookahead checks, as created or loaded (either pointer may be NULL). */
lacache_status lacache_get_config(const lacache_t* h, lacache_config* cfg, lacache_ensemble* ens);
lacache_status lacache_load(const char* path, int32_t device, int64_t capacity, lacache_t** out);

/* Decision counters of a handle (section 4.1's hit metrics count these outcomes): lookups and queries looked up,
 * and of those queries the HITs, lookahead rejections (REJECT) and key misses (MISS_KEY); entries inserted and
 * misses appended. */
typedef struct {
  int64_t lookups;
  int64_t queries;
  int64_t hits;
  int64_t rejects;
  int64_t key_misses;
  int64_t inserted;
  int64_t appended;
} lacache_stats;

/* The counters since create or the last reset (reset != 0 zeroes them after reading). Synchronizes the handle's
 * device: every lookup issued before the call is counted. Lookups through lacache_lookup_noalloc have no handle
 * and are not counted. */
lacache_status lacache_get_stats(lacache_t* h, lacache_stats* out, int32_t reset);

/* Number of stage-1 partial lists the last lookup used, and which stage-1 kernel it ran (lacache_stage1; a
 * tensor-core lookup reports LACACHE_STAGE1_TENSOR or LACACHE_STAGE1_TENSOR_PAIR). */
lacache_status lacache_last_launch(const lacache_t* h, int32_t* n_splits, int32_t* stage1_kernel);

/* Stage timing (measurement). lacache_stage_timing(h, m) with m > 0 makes the next m lookups record CUDA events
 * around their stage-1 and stage-2 kernels on the lookup's own stream (three cudaEventRecord calls per lookup;
 * the events are created here, not in the lookups). m = 0 turns it off and frees the events.
 * lacache_stage_times synchronizes on the last recorded event and returns, over the lookups timed since the
 * previous call, the summed device time of stage 1 (the key-check kernel) and of stage 2 (merge, lookahead
 * check and decision), and how many lookups were timed; it then restarts the count. */
lacache_status lacache_stage_timing(lacache_t* h, int32_t max_lookups);
lacache_status lacache_stage_times(lacache_t* h, double* stage1_ms, double* stage2_ms, int64_t* lookups);

/* Test support for failure detection. The next `lookups` lookups that run the tensor-core stage 1 make its first
 * CTA withhold one of its TMA loads: nothing is copied and nothing arrives on that pipeline stage, so the MMA
 * issuer's bounded wait (about one second) runs out. The kernel then records LACACHE_ERR_DEVICE_TIMEOUT, its other
 * roles stop, its issued copies and MMAs drain, TMEM is freed and it exits. The context stays usable: the next
 * lacache_sync reports the timeout and later lookups run normally. The affected lookup's outputs are undefined.
 * Lookups through the SimHash index take the injection when the popcount scan runs its shared-memory ring form
 * (512-bit signatures, or one query on a store of at least 16 tiles of 512 entries per split): its first CTA
 * withholds the bulk copy of its first tile, every thread's bounded wait for that tile runs out, the CTA still
 * ends its passes and waits (bounded) for its issued copies, and the timeout is recorded the same way.
 * On CTA pairs (B > 128) the first CTA is the leader of the first pair; its abort stops its peer too. A single
 * query tile (B <= 128) runs on a dynamic schedule: the stall happens only if the first CTA claims a key tile, which
 * is certain when the store holds many more 256-key tiles than the GPU has SMs. 0 cancels. */
lacache_status lacache_inject_stall(lacache_t* h, int32_t lookups);

/* Lookup that allocates nothing, for callers that cannot allocate device memory. Examples: a serving runtime or
 * framework whose allocator owns all device memory, code that must not trigger the device synchronization that
 * cudaMalloc and cudaFree can cause, and plug-ins with a fixed memory budget. The paper has no counterpart; this
 * is a deployment variant of lacache_lookup.
 *
 * It runs a single lookahead check (m = 1). The cache rows are caller-owned device arrays in the store's layout:
 * key_dev and prefix_dev [n x d] bf16
 * (16-byte aligned), ids_dev [n x k] int32. Queries and outputs are as for lacache_lookup. From *cfg it uses
 * d, k, tau_c, tau_a, top_c, token_match_min, check_mode, device and stage1; capacity and max_batch are ignored.
 * The stage-1 scratch lives in an 8 MiB file-scope device array of the library, which every GPU that loads the
 * library holds until the process exits. 512 bytes of it hold a status word and alignment padding, so a batch
 * fits only if B * (8 * top_c + 8) <= 8 MiB - 512 bytes (for top_c = 32, B <= 31773); larger batches return
 * LACACHE_ERR_UNSUPPORTED and nothing runs. stage1 = LACACHE_STAGE1_AUTO chooses as for a handle, and runs the
 * streaming scan if the driver offers no TMA descriptor encoder; an explicit LACACHE_STAGE1_TENSOR then gives
 * LACACHE_ERR_CUDA. The first call on a device does a one-time set-up (it looks up the
 * array's device address), so make that first call before any stream capture. All calls on a device share the
 * array: calls that overlap on the GPU (other streams, other host threads) race and give undefined results, so
 * issue them on one stream. A device-side timeout is not reported by this entry point (its outputs are then
 * undefined). Asynchronous on cuda_stream. */
lacache_status lacache_lookup_noalloc(const lacache_config* cfg, int64_t n, const void* key_dev,
                                      const void* prefix_dev, const int32_t* ids_dev, int32_t B,
                                      const void* q_emb_dev, const void* q_prefix_dev, const int32_t* q_ids_dev,
                                      const lacache_result* out, void* cuda_stream);

/* Threshold calibration (App. A.2, "Threshold Calibration"). For n benign pairs (x_i, y_i), bf16 rows of x_dev and
 * y_dev ([n x d] each, 16-byte aligned), writes sims_dev[i] = sim(x_i, y_i) (fp32 dot of unit vectors), then
 * result_dev[0] = the nearest-rank `percentile` of the sims (the value of rank ceil(percentile / 100 * n) in
 * ascending order, at least 1) and result_dev[1] = min(cap, result_dev[0]). The paper's rules are
 * tau_c = min(0.80, P5 of the query-pair sims) and tau_a = min(0.70, P10 of the response-prefix sims), the latter
 * per embedding model. sims_dev ([n] floats), result_dev (2 floats) and workspace_dev
 * (lacache_calibrate_workspace_bytes() bytes, 16-byte aligned, any contents) are caller device buffers; nothing is
 * allocated. Calls sharing a workspace must not overlap on the GPU. Asynchronous on cuda_stream. */
lacache_status lacache_calibrate(int64_t n, int32_t d, const void* x_dev, const void* y_dev, double percentile,
                                 float cap, float* sims_dev, float* result_dev, void* workspace_dev,
                                 void* cuda_stream);
size_t lacache_calibrate_workspace_bytes(void);

/* Reuse of the lookahead prefix on a miss (section 3.3, "Speculative Decoding"). A query that is not served has
 * its k draft tokens f_k(x) verified by the target model in one forward pass: from the first token on, draft token
 * t is accepted if P_f(t) >= P_g(t), and the first rejection hands decoding to the target model. Given
 * p_target_dev and p_draft_dev ([B x k] floats: each model's probability of each draft token), writes
 * accepted_dev[q] = the number of leading accepted tokens, or -1 where status_dev[q] == LACACHE_HIT (a served query
 * decodes nothing). status_dev may be NULL (every query verified). Asynchronous on cuda_stream. */
lacache_status lacache_verify_draft(int32_t B, int32_t k, const float* p_target_dev, const float* p_draft_dev,
                                    const uint8_t* status_dev, int32_t* accepted_dev, void* cuda_stream);

/* Static description of a status code. */
const char* lacache_status_string(lacache_status s);

/* Entry-range sharding (one store split across GPUs by row ranges; a multi-GPU form of the lookup). Each GPU
 * holds global entries [id_base, id_base + n) in its own handle and runs lacache_lookup on the same batch with the
 * candidate outputs (cand_id, cand_score, cand_prefix_score, cand_matches, cand_pass, and cand_prefix_scores for
 * an ensemble). The shards' outputs are then exchanged, for instance by one all-gather, and merged here into the
 * result of one lookup over the whole store.
 *
 * The merge is exact. The key check is per entry, so A_q is the union of the shards' sets. Every member of the
 * global candidate list C_q is among its own shard's first top_c, so C_q is the first top_c of the shards' lists
 * by (key score desc, global id asc). A candidate's lookahead result depends only on its own row. The served
 * entry is the first passing member of C_q. key_score on a miss is the maximum over the shards. All shards must
 * use the same top_c, thresholds and check mode.
 *
 * A shard's outputs as the merge reads them: device pointers on the current device, laid out as lacache_lookup
 * writes them. */
typedef struct {
  const int32_t* cand_id;            /* [B x top_c] local ids, -1 padded */
  const float* cand_score;           /* [B x top_c] */
  const float* cand_prefix_score;    /* [B x top_c] */
  const int32_t* cand_matches;       /* [B x top_c] */
  const uint8_t* cand_pass;          /* [B x top_c] */
  const float* cand_prefix_scores;   /* [B x top_c x m]; may be NULL when m == 1 (cand_prefix_score is used) */
  const float* key_score;            /* [B] */
  const int32_t* n_cand;             /* [B] */
  int64_t id_base;                   /* global id of the shard's entry 0; bases increase with the shard index */
} lacache_shard_result;

#define LACACHE_MAX_SHARDS 16

/* Merge the outputs of G shards (1..LACACHE_MAX_SHARDS; shards is a host array) for a batch of B queries into
 * *out (device pointers; the same fields and optional fields as a lookup; entry and candidate ids are global and
 * must fit in int32). m is the number of lookahead models (1 without an ensemble). Runs on the current device,
 * asynchronously on cuda_stream. */
lacache_status lacache_merge_shards(int32_t G, const lacache_shard_result* shards, int32_t B, int32_t top_c,
                                    int32_t m, const lacache_result* out, void* cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* LACACHE_H_ */
