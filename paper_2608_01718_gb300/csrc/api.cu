// C-ABI entry points of liblacache.so (declared in include/lacache.h): the device store, insert and the cache
// update of the serve loop, and the dispatch of a lookup to the stage-1 and stage-2 kernels.
#include <cuda.h>
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <new>

#include <algorithm>

#include "internal.cuh"

struct lacache {
  lacache_config cfg;
  lacache_ensemble ens;      // the lookahead checks (m = 1 for lacache_create)
  int pd;                    // prefix row length: sum of ens.dims
  int num_sms;
  int max_splits;
  int64_t n;                 // valid entries, as of the calls issued so far
  __nv_bfloat16* key;        // [capacity x d]
  __nv_bfloat16* prefix;     // [capacity x pd]
  int32_t* ids;              // [capacity x k]
  uint64_t* part_cand;       // [max_splits x max_batch x top_c]
  lc::PartMeta* part_meta;   // [max_splits x max_batch]
  unsigned int* dev_status;  // device status word
  int32_t* append_dst;       // [max_batch] destination rank of each appended query
  int32_t* append_count;     // device count of appended rows
  int32_t* append_count_host;  // pinned
  unsigned char* stage_in;   // device staging for lookup_host inputs: two slots, used in turn
  int stage_slot;            // the slot the next host lookup's inputs go to
  unsigned char* stage_out;  // device staging for lookup_host results
  unsigned char* stage_host; // pinned host staging of lookup_host results (mapped: the kernels write it directly)
  unsigned char* stage_host_dev; // device address of stage_host, or nullptr if the device cannot map it
  int last_splits;
  int last_kernel;
  lc::EncodeTiledFn encode;
  int inject_stall;          // lookups left that withhold one stage-1 load (failure-detection tests)
  int* tile_ctr;             // [next tile, CTAs done] of the dynamic stage-1 schedule (each launch leaves them zero)
  unsigned long long* counters;  // device: decisions [hits, rejects, key misses] (stage 2 adds per query)
  int64_t lookups, queries, inserted, appended;   // host-side counters
  int lsh_bits;              // SimHash index: signature bits (0 = no index)
  int lsh_radius;
  uint32_t* sig;             // [capacity x lsh_bits/32] entry signatures
  uint32_t* qsig;            // [max_batch x lsh_bits/32] query signatures of the current lookup
  __nv_bfloat16* hyper;      // [lsh_bits x d] hyperplanes
  uint8_t* sig_index;        // the signatures expanded for the tensor-core scan (lsh_index_bytes)
  cudaEvent_t* events;       // [3 x event_cap] stage-timing events, or NULL
  int event_cap;
  int event_used;
};

namespace {

using lc::Stage1Args;
using lc::Stage2Args;

class DeviceGuard {
 public:
  explicit DeviceGuard(int dev) {
    ok_ = cudaGetDevice(&prev_) == cudaSuccess;
    if (ok_ && prev_ != dev) ok_ = cudaSetDevice(dev) == cudaSuccess;
    dev_ = dev;
  }
  ~DeviceGuard() {
    if (ok_ && prev_ != dev_) cudaSetDevice(prev_);
  }
  bool ok() const { return ok_; }

 private:
  int prev_ = 0, dev_ = 0;
  bool ok_ = false;
};

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

lacache_status from_cuda(cudaError_t e) { return e == cudaSuccess ? LACACHE_OK : LACACHE_ERR_CUDA; }

// f32 -> bf16 (round to nearest even) of the key rows (count_a elements) and prefix rows (count_b), into the store.
__global__ void convert_rows_kernel(const float* __restrict__ a, const float* __restrict__ b,
                                    __nv_bfloat16* __restrict__ da, __nv_bfloat16* __restrict__ db, int64_t count_a,
                                    int64_t count_b) {
  const int64_t count = count_a > count_b ? count_a : count_b;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < count; i += (int64_t)gridDim.x * blockDim.x) {
    if (i < count_a) da[i] = __float2bfloat16_rn(a[i]);
    if (i < count_b) db[i] = __float2bfloat16_rn(b[i]);
  }
}

// Rank of every non-HIT query among the non-HIT queries of the batch (query order), and their count.
__global__ void append_rank_kernel(const uint8_t* __restrict__ status, int B, int32_t* __restrict__ dst,
                                   int32_t* __restrict__ count) {
  __shared__ int warp_tot[32];
  __shared__ int carry;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  for (int base = 0; base < B; base += blockDim.x) {
    const int q = base + threadIdx.x;
    const int flag = (q < B && status[q] != LACACHE_HIT) ? 1 : 0;
    const unsigned ballot = __ballot_sync(0xffffffffu, flag);
    const int in_warp = __popc(ballot & ((1u << lane) - 1u));
    if (lane == 0) warp_tot[warp] = __popc(ballot);
    __syncthreads();
    int before = carry;
    for (int w = 0; w < warp; ++w) before += warp_tot[w];
    if (q < B) dst[q] = flag ? before + in_warp : -1;
    __syncthreads();
    if (threadIdx.x == 0) {
      int t = 0;
      for (int w = 0; w < nw; ++w) t += warp_tot[w];
      carry += t;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) *count = carry;
}

// Copy the rows of the ranked queries into the store at n0 + rank, unless the batch would overflow capacity.
__global__ void append_rows_kernel(const uint4* __restrict__ q_emb, const uint4* __restrict__ q_pre,
                                   const int32_t* __restrict__ q_ids, const int32_t* __restrict__ dst,
                                   const int32_t* __restrict__ count, int B, int d, int pd, int k, int64_t n0,
                                   int64_t capacity, uint4* __restrict__ key, uint4* __restrict__ pre,
                                   int32_t* __restrict__ ids) {
  if (n0 + *count > capacity) return;
  const int kv = d / 8, pv = pd / 8;   // 16-byte vectors per key row and per prefix row
  const int q = blockIdx.x;
  if (q >= B) return;
  const int r = dst[q];
  if (r < 0) return;
  const int64_t row = n0 + r;
  for (int i = threadIdx.x; i < kv; i += blockDim.x) key[row * kv + i] = q_emb[(int64_t)q * kv + i];
  for (int i = threadIdx.x; i < pv; i += blockDim.x) pre[row * pv + i] = q_pre[(int64_t)q * pv + i];
  for (int i = threadIdx.x; i < k; i += blockDim.x) ids[row * k + i] = q_ids[(int64_t)q * k + i];
}

// lookup_host's inputs, read by the device straight from mapped pinned host memory (NVLink-C2C on Grace) into the
// device staging: one launch for the three arrays instead of one DMA copy each. Segments with zero bytes are
// skipped; 16-byte vectors where both ends are aligned, bytes otherwise.
// The kernel is a programmatic dependent of the previous lookup's stage 2, so it copies while that stage runs:
// host lookups use the two staging slots in turn, and the lookup that last used this slot (two host lookups back)
// has completed. Before it exits it waits for the grids before it, so its completion also means the previous
// lookup has ended (the stage-1 grid after it, which waits for it, then overwrites the partial lists the previous
// stage 2 read). Lets the stage-1 grid (a programmatic dependent too) start its set-up at once; that grid waits for
// this one before reading anything.
struct GatherSeg {
  const unsigned char* src;
  unsigned char* dst;
  size_t bytes;
};
struct GatherArgs {
  GatherSeg seg[3];
};
__global__ void gather_host_kernel(GatherArgs g) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const size_t tid = blockIdx.x * (size_t)blockDim.x + threadIdx.x, nth = (size_t)gridDim.x * blockDim.x;
  for (int s = 0; s < 3; ++s) {
    const GatherSeg e = g.seg[s];
    const bool vec = (((uintptr_t)e.src | (uintptr_t)e.dst) & 15u) == 0;
    const size_t nv = vec ? e.bytes / 16 : 0;
    const uint4* sv = reinterpret_cast<const uint4*>(e.src);
    uint4* dv = reinterpret_cast<uint4*>(e.dst);
    for (size_t i = tid; i < nv; i += nth) dv[i] = sv[i];
    for (size_t i = nv * 16 + tid; i < e.bytes; i += nth) e.dst[i] = e.src[i];
  }
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

// The address through which the current device can read host pointer p, or nullptr when it has none (pageable
// memory, or pinned memory not mapped for this device). Asked of the driver on every call, never cached: a
// device access through a stale answer would fault.
const void* mapped_device_pointer(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return a.type == cudaMemoryTypeHost ? a.devicePointer : nullptr;
}

// Output field p of an asynchronous host lookup as a device-writable address in *d: NULL stays NULL; anything else
// must be mapped pinned memory aligned to T.
template <typename T>
bool map_output(T* p, T** d) {
  *d = nullptr;
  if (!p) return true;
  if (reinterpret_cast<uintptr_t>(p) % alignof(T)) return false;
  *d = static_cast<T*>(const_cast<void*>(mapped_device_pointer(p)));
  return *d != nullptr;
}

// The three inputs of a host-buffer lookup (key embeddings, prefix embeddings, token ids): where they are, where
// they go in the handle's device staging, and their sizes.
struct HostInputs {
  const void* src[3];
  unsigned char* dst[3];
  size_t bytes[3];
};
size_t stage_in_bytes(const lacache_config& c, int pd);
// Distance between the two staging slots: a slot's bytes rounded up to 256, so that both slots' arrays keep the
// alignment the kernels and the TMA descriptors need (a slot ends with B * k * 4 bytes of token ids).
size_t stage_in_stride(const lacache_config& c, int pd) { return (stage_in_bytes(c, pd) + 255) & ~(size_t)255; }

// The inputs go to the handle's current staging slot; a host lookup that enqueues work then moves the handle to
// the other slot (next_stage_slot), so consecutive host lookups alternate.
HostInputs host_inputs(const lacache* h, int B, const void* emb, const void* pre, const int32_t* ids) {
  const lacache_config& c = h->cfg;
  HostInputs in{{emb, pre, ids}, {}, {(size_t)B * c.d * 2, (size_t)B * h->pd * 2, (size_t)B * c.k * 4}};
  in.dst[0] = h->stage_in + (size_t)h->stage_slot * stage_in_stride(c, h->pd);
  in.dst[1] = in.dst[0] + (size_t)c.max_batch * c.d * 2;
  in.dst[2] = in.dst[1] + (size_t)c.max_batch * h->pd * 2;
  return in;
}

void next_stage_slot(lacache* h) { h->stage_slot ^= 1; }

// One gather kernel for the segments of g, `bytes` in all (a programmatic dependent launch).
cudaError_t launch_gather(const lacache* h, const GatherArgs& g, size_t bytes, cudaStream_t st) {
  const size_t vec = (bytes + 15) / 16;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)std::min<size_t>((vec + 255) / 256, (size_t)2 * h->num_sms));
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gather_host_kernel, g);
}

// A handle set to the SimHash stage can look up only once its index is enabled.
bool lookup_ready(const lacache* h) { return h->cfg.stage1 != LACACHE_STAGE1_LSH || h->lsh_bits; }

size_t stage_in_bytes(const lacache_config& c, int pd) {
  return (size_t)c.max_batch * ((size_t)2 * c.d + (size_t)2 * pd + (size_t)4 * c.k);
}
size_t stage_out_bytes(const lacache_config& c, int m) {
  // five [B] 4-byte arrays, one [B] byte array, four [B x top_c] 4-byte arrays, one [B x top_c] byte array, one
  // [B x m] and one [B x top_c x m] 4-byte array, each rounded up to 16 bytes
  const size_t cm = (size_t)c.top_c * m;
  return (size_t)c.max_batch * (21 + (size_t)c.top_c * 17 + (size_t)m * 4 + cm * 4) + 13 * 16;
}

// Layout of the results of lookup_host in the staging buffer: the arrays of a B-query batch packed back to back,
// each 16-byte aligned; an optional array is present iff `want` asks for it.
lacache_result staged_result(unsigned char* base, int B, int top_c, int m, const lacache_result& want,
                             size_t* bytes) {
  unsigned char* p = base;
  auto take = [&](size_t n) {
    unsigned char* r = p;
    p += (n + 15) & ~(size_t)15;
    return r;
  };
  const size_t b = (size_t)B, bc = (size_t)B * top_c;
  lacache_result r;
  r.entry_id = (int32_t*)take(b * 4);
  r.key_score = (float*)take(b * 4);
  r.prefix_score = (float*)take(b * 4);
  r.token_matches = (int32_t*)take(b * 4);
  r.n_cand = (int32_t*)take(b * 4);
  r.status = (uint8_t*)take(b);
  r.cand_id = want.cand_id ? (int32_t*)take(bc * 4) : nullptr;
  r.cand_score = want.cand_score ? (float*)take(bc * 4) : nullptr;
  r.cand_prefix_score = want.cand_prefix_score ? (float*)take(bc * 4) : nullptr;
  r.cand_matches = want.cand_matches ? (int32_t*)take(bc * 4) : nullptr;
  r.prefix_scores = want.prefix_scores ? (float*)take(b * m * 4) : nullptr;
  r.cand_pass = want.cand_pass ? (uint8_t*)take(bc) : nullptr;
  r.cand_prefix_scores = want.cand_prefix_scores ? (float*)take(bc * m * 4) : nullptr;
  *bytes = (size_t)(p - base);
  return r;
}

void free_events(lacache* h) {
  if (!h->events) return;
  for (int i = 0; i < 3 * h->event_cap; ++i)
    if (h->events[i]) cudaEventDestroy(h->events[i]);
  free(h->events);
  h->events = nullptr;
  h->event_cap = h->event_used = 0;
}

void free_lsh(lacache* h) {
  cudaFree(h->sig);
  cudaFree(h->qsig);
  cudaFree(h->hyper);
  cudaFree(h->sig_index);
  h->sig = h->qsig = nullptr;
  h->hyper = nullptr;
  h->sig_index = nullptr;
  h->lsh_bits = 0;
}

// Signatures of store rows [first, first + n), packed and expanded, when the index is enabled.
cudaError_t sign_rows(lacache* h, int64_t first, int64_t n, cudaStream_t st) {
  if (!h->lsh_bits || n <= 0) return cudaSuccess;
  const int words = h->lsh_bits / 32;
  cudaError_t e = lc::launch_signatures(h->key + first * h->cfg.d, n, h->cfg.d, h->hyper, h->lsh_bits,
                                        h->sig + first * words, h->dev_status, h->encode, h->num_sms, st);
  if (e == cudaSuccess && h->sig_index)
    e = lc::launch_expand_signatures(h->sig, first, n, h->lsh_bits, h->sig_index, h->num_sms, st);
  return e;
}

void free_all(lacache* h) {
  free_lsh(h);
  free_events(h);
  cudaFree(h->key);
  cudaFree(h->prefix);
  cudaFree(h->ids);
  cudaFree(h->part_cand);
  cudaFree(h->part_meta);
  cudaFree(h->dev_status);
  cudaFree(h->append_dst);
  cudaFree(h->append_count);
  cudaFree(h->tile_ctr);
  cudaFree(h->counters);
  cudaFree(h->stage_in);
  cudaFree(h->stage_out);
  if (h->append_count_host) cudaFreeHost(h->append_count_host);
  if (h->stage_host) cudaFreeHost(h->stage_host);
}

// gathered: the queries were just written by gather_host_kernel, so the first kernel waits for it before reading.
lacache_status run_lookup(lacache* h, int32_t B, const void* q_emb, const void* q_prefix, const int32_t* q_ids,
                          const lacache_result& out, cudaStream_t st, bool gathered = false) {
  const lacache_config& c = h->cfg;
  if (!lookup_ready(h)) return LACACHE_ERR_INVALID_ARG;
  int splits = 0;
  int kernel = 0;
  cudaEvent_t* ev = nullptr;
  if (h->events && h->event_used < h->event_cap) ev = h->events + 3 * h->event_used++;
  if (ev && cudaEventRecord(ev[0], st) != cudaSuccess) return LACACHE_ERR_CUDA;
  if (h->n > 0) {
    Stage1Args a{};
    a.keys = h->key;
    a.n = h->n;
    a.d = c.d;
    a.q = reinterpret_cast<const __nv_bfloat16*>(q_emb);
    a.B = B;
    a.tau_c = c.tau_c;
    a.top_c = c.top_c;
    a.part_cand = h->part_cand;
    a.part_meta = h->part_meta;
    a.dev_status = h->dev_status;
    a.inputs_from_previous = gathered ? 1 : 0;
    kernel = c.stage1 == LACACHE_STAGE1_AUTO ? lc::auto_stage1(h->n, c.d, B) : c.stage1;
    if (h->inject_stall > 0 && kernel == LACACHE_STAGE1_TENSOR) {
      a.inject_stall = 1;
      --h->inject_stall;
    }
    // the SimHash scan takes the injection only in its ring form (the launcher reports which form ran)
    if (h->inject_stall > 0 && kernel == LACACHE_STAGE1_LSH) a.inject_stall = 1;
    cudaError_t e;
    if (kernel == LACACHE_STAGE1_TENSOR) {
      if (!h->encode) return LACACHE_ERR_CUDA;
      // the kernel leaves the schedule's counters zero for the next launch (the previous one has completed
      // before this one touches memory)
      a.tile_ctr = h->tile_ctr;
      bool paired = false;
      e = lc::launch_stage1_tensor(a, h->encode, h->num_sms, h->max_splits, st, &splits, &paired);
      if (paired) kernel = LACACHE_STAGE1_TENSOR_PAIR;
    } else if (kernel == LACACHE_STAGE1_LSH) {
      // batches of up to kSignCudaCoreMaxBatch queries are signed on the CUDA cores (one CTA per query and word,
      // about one memory round trip), larger ones by the tensor-core GEMM that signs the entries: the CUDA-core
      // kernel reads each 32-hyperplane block once per query, which costs more than the GEMM beyond that
      e = B > lc::kSignCudaCoreMaxBatch
              ? lc::launch_signatures(a.q, B, c.d, h->hyper, h->lsh_bits, h->qsig, h->dev_status, h->encode,
                                      h->num_sms, st, gathered)
              : lc::launch_sign_queries(a.q, B, c.d, h->hyper, h->lsh_bits, h->qsig, st, gathered);
      if (e == cudaSuccess) {
        lc::LshArgs l{h->sig, h->qsig, h->lsh_bits / 32, h->lsh_radius, h->sig_index};
        if (B >= lc::lsh_tensor_min_batch(h->lsh_bits) && h->sig_index) {
          e = lc::launch_stage1_lsh_tc(a, l, h->num_sms, h->max_splits, st, &splits);
          kernel = LACACHE_STAGE1_LSH_TENSOR;
        } else {
          bool ring = false;
          e = lc::launch_stage1_lsh(a, l, h->num_sms, h->max_splits, st, &splits, &ring);
          if (ring && a.inject_stall) --h->inject_stall;
        }
      }
    } else {
      e = lc::launch_stage1_stream(a, h->num_sms, h->max_splits, st, &splits);
    }
    if (e != cudaSuccess) return LACACHE_ERR_CUDA;
  }
  Stage2Args b{};
  b.n = h->n;
  b.part_cand = h->part_cand;
  b.part_meta = h->part_meta;
  b.splits = splits;
  b.B = B;
  b.pd = h->pd;
  b.k = c.k;
  b.top_c = c.top_c;
  b.m = h->ens.m;
  for (int i = 0; i < h->ens.m; ++i) {
    b.seg[i + 1] = b.seg[i] + h->ens.dims[i];
    b.tau_m[i] = h->ens.tau_a[i];
  }
  b.check_mode = c.check_mode;
  b.token_match_min = c.token_match_min;
  b.prefix = h->prefix;
  b.ids = h->ids;
  b.q_prefix = reinterpret_cast<const __nv_bfloat16*>(q_prefix);
  b.q_ids = q_ids;
  b.out = out;
  b.counters = h->counters;
  if (ev && cudaEventRecord(ev[1], st) != cudaSuccess) return LACACHE_ERR_CUDA;
  if (lc::launch_stage2(b, st) != cudaSuccess) return LACACHE_ERR_CUDA;
  if (ev && cudaEventRecord(ev[2], st) != cudaSuccess) return LACACHE_ERR_CUDA;
  h->last_splits = splits;
  h->last_kernel = kernel;
  ++h->lookups;
  h->queries += B;
  return LACACHE_OK;
}

bool result_ok(const lacache_result* r) {
  return r && r->entry_id && r->status && r->key_score && r->prefix_score && r->token_matches && r->n_cand;
}

}  // namespace

extern "C" {

const char* lacache_status_string(lacache_status s) {
  switch (s) {
    case LACACHE_OK: return "ok";
    case LACACHE_ERR_INVALID_ARG: return "invalid argument";
    case LACACHE_ERR_CAPACITY: return "capacity exceeded";
    case LACACHE_ERR_OOM: return "device out of memory";
    case LACACHE_ERR_CUDA: return "CUDA error";
    case LACACHE_ERR_DEVICE_TIMEOUT: return "device wait timed out";
    case LACACHE_ERR_UNSUPPORTED: return "unsupported configuration";
    case LACACHE_ERR_IO: return "i/o error";
  }
  return "unknown status";
}

lacache_status lacache_create(const lacache_config* cfg, lacache_t** out) {
  if (!out) return LACACHE_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg) return LACACHE_ERR_INVALID_ARG;
  lacache_ensemble one;
  memset(&one, 0, sizeof(one));
  one.m = 1;
  one.dims[0] = cfg->d;
  one.tau_a[0] = cfg->tau_a;
  return lacache_create_ensemble(cfg, &one, out);
}

lacache_status lacache_create_ensemble(const lacache_config* cfg, const lacache_ensemble* ens, lacache_t** out) {
  if (!out) return LACACHE_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg || !ens) return LACACHE_ERR_INVALID_ARG;
  const lacache_config c = *cfg;
  if (ens->m < 1 || ens->m > LACACHE_MAX_MODELS) return LACACHE_ERR_INVALID_ARG;
  int pd = 0;
  for (int i = 0; i < ens->m; ++i) {
    if (ens->dims[i] <= 0 || isnan(ens->tau_a[i])) return LACACHE_ERR_INVALID_ARG;
    if (ens->dims[i] % 8 != 0) return LACACHE_ERR_UNSUPPORTED;
    pd += ens->dims[i];
  }
  if (pd > lc::kMaxD) return LACACHE_ERR_UNSUPPORTED;
  if (c.d <= 0 || c.k <= 0 || c.capacity <= 0 || c.top_c <= 0 || c.max_batch <= 0) return LACACHE_ERR_INVALID_ARG;
  if (isnan(c.tau_c) || isnan(c.tau_a)) return LACACHE_ERR_INVALID_ARG;
  if (c.check_mode < LACACHE_CHECK_EMB || c.check_mode > LACACHE_CHECK_BOTH) return LACACHE_ERR_INVALID_ARG;
  if (c.stage1 < LACACHE_STAGE1_AUTO || c.stage1 > LACACHE_STAGE1_LSH) return LACACHE_ERR_INVALID_ARG;
  if (c.token_match_min > c.k) return LACACHE_ERR_INVALID_ARG;
  if (c.d % 8 != 0 || c.d > lc::kMaxD || c.k > lc::kMaxK || c.top_c > lc::kMaxTopC) return LACACHE_ERR_UNSUPPORTED;
  if (c.capacity > (int64_t)INT32_MAX || c.max_batch > (1 << 20)) return LACACHE_ERR_UNSUPPORTED;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess) return LACACHE_ERR_CUDA;
  if (c.device < 0 || c.device >= ndev) return LACACHE_ERR_INVALID_ARG;
  DeviceGuard guard(c.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;

  lacache* h = new (std::nothrow) lacache;
  if (!h) return LACACHE_ERR_OOM;
  memset(h, 0, sizeof(*h));
  h->cfg = c;
  h->ens = *ens;
  h->pd = pd;
  if (cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, c.device) != cudaSuccess) {
    delete h;
    return LACACHE_ERR_CUDA;
  }
  h->max_splits = lc::max_splits_for(h->num_sms, c.max_batch, c.top_c);
  const size_t cap = (size_t)c.capacity;
  bool ok = cudaMalloc(&h->key, cap * c.d * 2) == cudaSuccess &&
            cudaMalloc(&h->prefix, cap * pd * 2) == cudaSuccess &&
            cudaMalloc(&h->ids, cap * c.k * 4) == cudaSuccess &&
            cudaMalloc(&h->part_cand, (size_t)h->max_splits * c.max_batch * c.top_c * 8) == cudaSuccess &&
            cudaMalloc(&h->part_meta, (size_t)h->max_splits * c.max_batch * sizeof(lc::PartMeta)) == cudaSuccess &&
            cudaMalloc(&h->dev_status, 4) == cudaSuccess &&
            cudaMalloc(&h->append_dst, (size_t)c.max_batch * 4) == cudaSuccess &&
            cudaMalloc(&h->append_count, 4) == cudaSuccess &&
            cudaMalloc(&h->tile_ctr, 2 * sizeof(int)) == cudaSuccess &&
            cudaMalloc(&h->counters, 3 * sizeof(unsigned long long)) == cudaSuccess &&
            cudaMemset(h->counters, 0, 3 * sizeof(unsigned long long)) == cudaSuccess &&
            cudaMemset(h->tile_ctr, 0, 2 * sizeof(int)) == cudaSuccess &&
            cudaMalloc(&h->stage_in, 2 * stage_in_stride(c, pd)) == cudaSuccess &&
            cudaMalloc(&h->stage_out, stage_out_bytes(c, ens->m)) == cudaSuccess &&
            cudaMallocHost(&h->append_count_host, 4) == cudaSuccess &&
            cudaHostAlloc((void**)&h->stage_host, stage_out_bytes(c, ens->m), cudaHostAllocMapped) == cudaSuccess &&
            cudaMemset(h->dev_status, 0, 4) == cudaSuccess &&
            cudaMemset(h->part_cand, 0, (size_t)h->max_splits * c.max_batch * c.top_c * 8) == cudaSuccess &&
            cudaDeviceSynchronize() == cudaSuccess;
  if (!ok) {
    cudaGetLastError();
    free_all(h);
    delete h;
    return LACACHE_ERR_OOM;
  }
  if (cudaHostGetDevicePointer((void**)&h->stage_host_dev, h->stage_host, 0) != cudaSuccess) {
    cudaGetLastError();
    h->stage_host_dev = nullptr;   // results then come back with one device-to-host copy
  }
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
          cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    h->encode = reinterpret_cast<lc::EncodeTiledFn>(fn);
  *out = h;
  return LACACHE_OK;
}

lacache_status lacache_destroy(lacache_t* h) {
  if (!h) return LACACHE_OK;
  DeviceGuard guard(h->cfg.device);
  cudaDeviceSynchronize();
  free_all(h);
  delete h;
  return LACACHE_OK;
}

lacache_status lacache_insert(lacache_t* h, int64_t n, const void* key_dev, const void* prefix_dev,
                              const int32_t* ids_dev, int32_t dtype, int64_t* first_id, void* cuda_stream) {
  lc::NvtxRange nvtx("lacache_insert");
  if (!h || n < 0) return LACACHE_ERR_INVALID_ARG;
  if (dtype != LACACHE_BF16 && dtype != LACACHE_F32) return LACACHE_ERR_INVALID_ARG;
  if (n > 0 && (!key_dev || !prefix_dev || !ids_dev)) return LACACHE_ERR_INVALID_ARG;
  if (n > h->cfg.capacity - h->n) return LACACHE_ERR_CAPACITY;
  if (first_id) *first_id = h->n;
  if (n == 0) return LACACHE_OK;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  const int d = h->cfg.d, k = h->cfg.k, pd = h->pd;
  __nv_bfloat16* kdst = h->key + h->n * d;
  __nv_bfloat16* pdst = h->prefix + h->n * pd;
  cudaError_t e;
  if (dtype == LACACHE_BF16) {
    e = cudaMemcpyAsync(kdst, key_dev, (size_t)n * d * 2, cudaMemcpyDeviceToDevice, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(pdst, prefix_dev, (size_t)n * pd * 2, cudaMemcpyDeviceToDevice, st);
  } else {
    const int64_t count = n * (d > pd ? d : pd);
    const int threads = 256;
    const int64_t want = (count + threads - 1) / threads;
    const int blocks = (int)(want < (int64_t)h->num_sms * 32 ? want : (int64_t)h->num_sms * 32);
    convert_rows_kernel<<<blocks, threads, 0, st>>>((const float*)key_dev, (const float*)prefix_dev, kdst, pdst,
                                                    n * d, n * pd);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(h->ids + h->n * k, ids_dev, (size_t)n * k * 4, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess) e = sign_rows(h, h->n, n, st);
  if (e != cudaSuccess) return LACACHE_ERR_CUDA;
  h->n += n;
  h->inserted += n;
  return LACACHE_OK;
}

lacache_status lacache_lookup(lacache_t* h, int32_t B, const void* q_emb_dev, const void* q_prefix_dev,
                              const int32_t* q_ids_dev, const lacache_result* out, void* cuda_stream) {
  lc::NvtxRange nvtx("lacache_lookup");
  if (!h || B < 1 || B > h->cfg.max_batch) return LACACHE_ERR_INVALID_ARG;
  if (!q_emb_dev || !q_prefix_dev || !q_ids_dev || !result_ok(out)) return LACACHE_ERR_INVALID_ARG;
  if (!aligned16(q_emb_dev) || !aligned16(q_prefix_dev)) return LACACHE_ERR_INVALID_ARG;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  return run_lookup(h, B, q_emb_dev, q_prefix_dev, q_ids_dev, *out, (cudaStream_t)cuda_stream);
}

lacache_status lacache_lookup_host(lacache_t* h, int32_t B, const void* q_emb_host, const void* q_prefix_host,
                                   const int32_t* q_ids_host, const lacache_result* out_host, void* cuda_stream) {
  lc::NvtxRange nvtx("lacache_lookup_host");
  if (!h || B < 1 || B > h->cfg.max_batch) return LACACHE_ERR_INVALID_ARG;
  if (!q_emb_host || !q_prefix_host || !q_ids_host || !result_ok(out_host)) return LACACHE_ERR_INVALID_ARG;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  if (!lookup_ready(h)) return LACACHE_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  const lacache_config& c = h->cfg;
  const HostInputs in = host_inputs(h, B, q_emb_host, q_prefix_host, q_ids_host);
  next_stage_slot(h);
  // Inputs: arrays in mapped pinned memory are gathered by one kernel; any other array is copied by DMA.
  GatherArgs g{};
  size_t gathered = 0;
  for (int i = 0; i < 3; ++i) {
    const void* dev_src = mapped_device_pointer(in.src[i]);
    if (dev_src) {
      g.seg[i] = GatherSeg{static_cast<const unsigned char*>(dev_src), in.dst[i], in.bytes[i]};
      gathered += in.bytes[i];
    } else if (cudaMemcpyAsync(in.dst[i], in.src[i], in.bytes[i], cudaMemcpyHostToDevice, st) != cudaSuccess) {
      return LACACHE_ERR_CUDA;
    }
  }
  if (gathered && launch_gather(h, g, gathered, st) != cudaSuccess) return LACACHE_ERR_CUDA;
  size_t bytes = 0;
  // Results: written by the kernels straight into the mapped pinned staging when the device can map it.
  unsigned char* out_stage = h->stage_host_dev ? h->stage_host_dev : h->stage_out;
  lacache_result dev = staged_result(out_stage, B, c.top_c, h->ens.m, *out_host, &bytes);
  lacache_result host = staged_result(h->stage_host, B, c.top_c, h->ens.m, *out_host, &bytes);
  lacache_status s =
      run_lookup(h, B, in.dst[0], in.dst[1], reinterpret_cast<const int32_t*>(in.dst[2]), dev, st, gathered != 0);
  if (s != LACACHE_OK) return s;
  if (!h->stage_host_dev &&
      cudaMemcpyAsync(h->stage_host, h->stage_out, bytes, cudaMemcpyDeviceToHost, st) != cudaSuccess)
    return LACACHE_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return LACACHE_ERR_CUDA;
  const size_t b4 = (size_t)B * 4, bc4 = (size_t)B * c.top_c * 4;
  struct Copy {
    void* dst;
    const void* src;
    size_t bytes;
  } copies[] = {
      {out_host->entry_id, host.entry_id, b4},         {out_host->status, host.status, (size_t)B},
      {out_host->key_score, host.key_score, b4},       {out_host->prefix_score, host.prefix_score, b4},
      {out_host->token_matches, host.token_matches, b4}, {out_host->n_cand, host.n_cand, b4},
      {out_host->cand_id, host.cand_id, bc4},          {out_host->cand_score, host.cand_score, bc4},
      {out_host->cand_prefix_score, host.cand_prefix_score, bc4}, {out_host->cand_matches, host.cand_matches, bc4},
      {out_host->prefix_scores, host.prefix_scores, b4 * h->ens.m},
      {out_host->cand_pass, host.cand_pass, (size_t)B * c.top_c},
      {out_host->cand_prefix_scores, host.cand_prefix_scores, bc4 * h->ens.m},
  };
  for (const Copy& cp : copies)
    if (cp.dst && cp.src) memcpy(cp.dst, cp.src, cp.bytes);
  return LACACHE_OK;
}

lacache_status lacache_lookup_host_async(lacache_t* h, int32_t B, const void* q_emb_host, const void* q_prefix_host,
                                         const int32_t* q_ids_host, const lacache_result* out_host,
                                         void* cuda_stream) {
  lc::NvtxRange nvtx("lacache_lookup_host_async");
  if (!h || B < 1 || B > h->cfg.max_batch) return LACACHE_ERR_INVALID_ARG;
  if (!q_emb_host || !q_prefix_host || !q_ids_host || !result_ok(out_host)) return LACACHE_ERR_INVALID_ARG;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  if (!lookup_ready(h)) return LACACHE_ERR_INVALID_ARG;
  // every address is checked before anything is enqueued
  const HostInputs in = host_inputs(h, B, q_emb_host, q_prefix_host, q_ids_host);
  GatherArgs g{};
  size_t gathered = 0;
  for (int i = 0; i < 3; ++i) {
    const void* dev_src = mapped_device_pointer(in.src[i]);
    if (!dev_src) return LACACHE_ERR_INVALID_ARG;
    g.seg[i] = GatherSeg{static_cast<const unsigned char*>(dev_src), in.dst[i], in.bytes[i]};
    gathered += in.bytes[i];
  }
  const lacache_result& o = *out_host;
  lacache_result dev{};
  const bool mapped = map_output(o.entry_id, &dev.entry_id) && map_output(o.status, &dev.status) &&
                      map_output(o.key_score, &dev.key_score) && map_output(o.prefix_score, &dev.prefix_score) &&
                      map_output(o.token_matches, &dev.token_matches) && map_output(o.n_cand, &dev.n_cand) &&
                      map_output(o.cand_id, &dev.cand_id) && map_output(o.cand_score, &dev.cand_score) &&
                      map_output(o.cand_prefix_score, &dev.cand_prefix_score) &&
                      map_output(o.cand_matches, &dev.cand_matches) &&
                      map_output(o.prefix_scores, &dev.prefix_scores) && map_output(o.cand_pass, &dev.cand_pass) &&
                      map_output(o.cand_prefix_scores, &dev.cand_prefix_scores);
  if (!mapped) return LACACHE_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  next_stage_slot(h);
  if (launch_gather(h, g, gathered, st) != cudaSuccess) return LACACHE_ERR_CUDA;
  return run_lookup(h, B, in.dst[0], in.dst[1], reinterpret_cast<const int32_t*>(in.dst[2]), dev, st, true);
}

lacache_status lacache_append_misses(lacache_t* h, int32_t B, const void* q_emb_dev, const void* q_prefix_dev,
                                     const int32_t* q_ids_dev, const uint8_t* status_dev, int64_t* first_id,
                                     int64_t* n_appended, void* cuda_stream) {
  lc::NvtxRange nvtx("lacache_append_misses");
  if (!h || B < 1 || B > h->cfg.max_batch) return LACACHE_ERR_INVALID_ARG;
  if (!q_emb_dev || !q_prefix_dev || !q_ids_dev || !status_dev) return LACACHE_ERR_INVALID_ARG;
  if (!aligned16(q_emb_dev) || !aligned16(q_prefix_dev)) return LACACHE_ERR_INVALID_ARG;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  const lacache_config& c = h->cfg;
  append_rank_kernel<<<1, 1024, 0, st>>>(status_dev, B, h->append_dst, h->append_count);
  append_rows_kernel<<<B, 128, 0, st>>>((const uint4*)q_emb_dev, (const uint4*)q_prefix_dev, q_ids_dev,
                                        h->append_dst, h->append_count, B, c.d, h->pd, c.k, h->n, c.capacity,
                                        (uint4*)h->key, (uint4*)h->prefix, h->ids);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(h->append_count_host, h->append_count, 4, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return LACACHE_ERR_CUDA;
  const int64_t m = *h->append_count_host;
  if (h->n + m > c.capacity) return LACACHE_ERR_CAPACITY;
  if (sign_rows(h, h->n, m, st) != cudaSuccess) return LACACHE_ERR_CUDA;
  if (first_id) *first_id = h->n;
  if (n_appended) *n_appended = m;
  h->n += m;
  h->appended += m;
  return LACACHE_OK;
}

lacache_status lacache_enable_lsh(lacache_t* h, int32_t bits, int32_t radius, const void* hyperplanes_dev,
                                  void* cuda_stream) {
  lc::NvtxRange nvtx("lacache_enable_lsh");
  if (!h || !hyperplanes_dev || ((uintptr_t)hyperplanes_dev & 15u)) return LACACHE_ERR_INVALID_ARG;
  if (bits != 128 && bits != 256 && bits != 512) return LACACHE_ERR_UNSUPPORTED;
  if (radius < 0 || radius > bits) return LACACHE_ERR_INVALID_ARG;
  if (!h->encode) return LACACHE_ERR_CUDA;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  if (h->lsh_bits && cudaStreamSynchronize(st) != cudaSuccess) return LACACHE_ERR_CUDA;
  free_lsh(h);
  const int words = bits / 32;
  const lacache_config& c = h->cfg;
  // the expanded copy only where batches can be large enough to use it
  const size_t index_bytes =
      c.max_batch >= lc::lsh_tensor_min_batch(bits) ? lc::lsh_index_bytes(c.capacity, bits) : 0;
  if (cudaMalloc(&h->sig, (size_t)c.capacity * words * 4) != cudaSuccess ||
      cudaMalloc(&h->qsig, (size_t)c.max_batch * words * 4) != cudaSuccess ||
      cudaMalloc(&h->hyper, (size_t)bits * c.d * 2) != cudaSuccess ||
      (index_bytes && cudaMalloc(&h->sig_index, index_bytes) != cudaSuccess)) {
    cudaGetLastError();
    free_lsh(h);
    return LACACHE_ERR_OOM;
  }
  // rows past the valid entries of the last block are read by the scan (and never used): keep them defined
  if (index_bytes && cudaMemsetAsync(h->sig_index, 0, index_bytes, st) != cudaSuccess) return LACACHE_ERR_CUDA;
  h->lsh_bits = bits;
  h->lsh_radius = radius;
  if (cudaMemcpyAsync(h->hyper, hyperplanes_dev, (size_t)bits * c.d * 2, cudaMemcpyDeviceToDevice, st) !=
          cudaSuccess ||
      sign_rows(h, 0, h->n, st) != cudaSuccess)
    return LACACHE_ERR_CUDA;
  return LACACHE_OK;
}

lacache_status lacache_read_signatures(const lacache_t* h, int64_t first, int64_t n, uint32_t* sig_dev,
                                       void* cuda_stream) {
  if (!h || !h->lsh_bits || !sig_dev || first < 0 || n < 0 || first + n > h->n) return LACACHE_ERR_INVALID_ARG;
  if (n == 0) return LACACHE_OK;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  const int words = h->lsh_bits / 32;
  return from_cuda(cudaMemcpyAsync(sig_dev, h->sig + first * words, (size_t)n * words * 4, cudaMemcpyDeviceToDevice,
                                   (cudaStream_t)cuda_stream));
}

lacache_status lacache_read_rows(const lacache_t* h, int64_t first, int64_t n, void* key_dev, void* prefix_dev,
                                 int32_t* ids_dev, void* cuda_stream) {
  if (!h || first < 0 || n < 0 || first + n > h->n) return LACACHE_ERR_INVALID_ARG;
  if (n == 0) return LACACHE_OK;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  const int d = h->cfg.d, k = h->cfg.k, pd = h->pd;
  cudaError_t e = cudaSuccess;
  if (key_dev) e = cudaMemcpyAsync(key_dev, h->key + first * d, (size_t)n * d * 2, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess && prefix_dev)
    e = cudaMemcpyAsync(prefix_dev, h->prefix + first * pd, (size_t)n * pd * 2, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess && ids_dev)
    e = cudaMemcpyAsync(ids_dev, h->ids + first * k, (size_t)n * k * 4, cudaMemcpyDeviceToDevice, st);
  return from_cuda(e);
}

lacache_status lacache_size(const lacache_t* h, int64_t* n) {
  if (!h || !n) return LACACHE_ERR_INVALID_ARG;
  *n = h->n;
  return LACACHE_OK;
}

lacache_status lacache_sync(lacache_t* h) {
  if (!h) return LACACHE_ERR_INVALID_ARG;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  if (cudaDeviceSynchronize() != cudaSuccess) return LACACHE_ERR_CUDA;
  unsigned int word = 0;
  if (cudaMemcpy(&word, h->dev_status, 4, cudaMemcpyDeviceToHost) != cudaSuccess) return LACACHE_ERR_CUDA;
  if (word && cudaMemset(h->dev_status, 0, 4) != cudaSuccess) return LACACHE_ERR_CUDA;
  return (word & lc::kDevTimeout) ? LACACHE_ERR_DEVICE_TIMEOUT : LACACHE_OK;
}

lacache_status lacache_stage_timing(lacache_t* h, int32_t max_lookups) {
  if (!h || max_lookups < 0) return LACACHE_ERR_INVALID_ARG;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  if (h->events) cudaDeviceSynchronize();
  free_events(h);
  if (max_lookups == 0) return LACACHE_OK;
  h->events = static_cast<cudaEvent_t*>(calloc((size_t)3 * max_lookups, sizeof(cudaEvent_t)));
  if (!h->events) return LACACHE_ERR_OOM;
  h->event_cap = max_lookups;
  for (int i = 0; i < 3 * max_lookups; ++i) {
    if (cudaEventCreate(&h->events[i]) != cudaSuccess) {
      free_events(h);
      return LACACHE_ERR_CUDA;
    }
  }
  return LACACHE_OK;
}

lacache_status lacache_stage_times(lacache_t* h, double* stage1_ms, double* stage2_ms, int64_t* lookups) {
  if (!h) return LACACHE_ERR_INVALID_ARG;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  double t1 = 0, t2 = 0;
  const int used = h->events ? h->event_used : 0;
  if (used && cudaEventSynchronize(h->events[3 * used - 1]) != cudaSuccess) return LACACHE_ERR_CUDA;
  for (int i = 0; i < used; ++i) {
    float a = 0, b = 0;
    if (cudaEventElapsedTime(&a, h->events[3 * i], h->events[3 * i + 1]) != cudaSuccess ||
        cudaEventElapsedTime(&b, h->events[3 * i + 1], h->events[3 * i + 2]) != cudaSuccess)
      return LACACHE_ERR_CUDA;
    t1 += a;
    t2 += b;
  }
  if (h->events) h->event_used = 0;
  if (stage1_ms) *stage1_ms = t1;
  if (stage2_ms) *stage2_ms = t2;
  if (lookups) *lookups = used;
  return LACACHE_OK;
}

lacache_status lacache_inject_stall(lacache_t* h, int32_t lookups) {
  if (!h || lookups < 0) return LACACHE_ERR_INVALID_ARG;
  h->inject_stall = lookups;
  return LACACHE_OK;
}

}  // extern "C"

namespace {

// Saved-cache file header (little-endian, fixed-width fields; padding is written as zeros).
constexpr char kFileMagic[8] = {'L', 'A', 'C', 'A', 'C', 'H', 'E', '1'};
constexpr uint32_t kFileVersion = 1;
struct FileHeader {
  char magic[8];
  uint32_t version;
  uint32_t header_bytes;
  lacache_config cfg;
  lacache_ensemble ens;
  int64_t n;
};
constexpr size_t kIoChunk = (size_t)64 << 20;   // bytes per staged copy

// Copies `bytes` between a device array and a file through a pinned staging buffer of at most kIoChunk bytes.
bool copy_out(FILE* f, const void* dev, size_t bytes, unsigned char* stage) {
  for (size_t off = 0; off < bytes; off += kIoChunk) {
    const size_t len = bytes - off < kIoChunk ? bytes - off : kIoChunk;
    if (cudaMemcpy(stage, static_cast<const unsigned char*>(dev) + off, len, cudaMemcpyDeviceToHost) != cudaSuccess ||
        fwrite(stage, 1, len, f) != len)
      return false;
  }
  return true;
}
bool copy_in(FILE* f, void* dev, size_t bytes, unsigned char* stage) {
  for (size_t off = 0; off < bytes; off += kIoChunk) {
    const size_t len = bytes - off < kIoChunk ? bytes - off : kIoChunk;
    if (fread(stage, 1, len, f) != len ||
        cudaMemcpy(static_cast<unsigned char*>(dev) + off, stage, len, cudaMemcpyHostToDevice) != cudaSuccess)
      return false;
  }
  return true;
}

}  // namespace

extern "C" {

lacache_status lacache_save(lacache_t* h, const char* path) {
  lc::NvtxRange nvtx("lacache_save");
  if (!h || !path) return LACACHE_ERR_INVALID_ARG;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok() || cudaDeviceSynchronize() != cudaSuccess) return LACACHE_ERR_CUDA;
  FileHeader hdr;
  memset(&hdr, 0, sizeof hdr);
  memcpy(hdr.magic, kFileMagic, sizeof kFileMagic);
  hdr.version = kFileVersion;
  hdr.header_bytes = (uint32_t)sizeof hdr;
  hdr.cfg = h->cfg;
  hdr.ens = h->ens;
  hdr.n = h->n;
  FILE* f = fopen(path, "wb");
  if (!f) return LACACHE_ERR_IO;
  const size_t n = (size_t)h->n;
  const size_t sizes[3] = {n * h->cfg.d * 2, n * h->pd * 2, n * h->cfg.k * 4};
  unsigned char* stage = nullptr;
  lacache_status s = LACACHE_OK;
  if (cudaMallocHost(&stage, kIoChunk) != cudaSuccess) {
    cudaGetLastError();
    s = LACACHE_ERR_OOM;
  } else if (fwrite(&hdr, 1, sizeof hdr, f) != sizeof hdr || !copy_out(f, h->key, sizes[0], stage) ||
             !copy_out(f, h->prefix, sizes[1], stage) || !copy_out(f, h->ids, sizes[2], stage)) {
    s = LACACHE_ERR_IO;
  }
  if (stage) cudaFreeHost(stage);
  if (fclose(f) != 0 && s == LACACHE_OK) s = LACACHE_ERR_IO;
  return s;
}

lacache_status lacache_get_config(const lacache_t* h, lacache_config* cfg, lacache_ensemble* ens) {
  if (!h) return LACACHE_ERR_INVALID_ARG;
  if (cfg) *cfg = h->cfg;
  if (ens) *ens = h->ens;
  return LACACHE_OK;
}

lacache_status lacache_load(const char* path, int32_t device, int64_t capacity, lacache_t** out) {
  lc::NvtxRange nvtx("lacache_load");
  if (!out) return LACACHE_ERR_INVALID_ARG;
  *out = nullptr;
  if (!path || capacity < 0) return LACACHE_ERR_INVALID_ARG;
  FILE* f = fopen(path, "rb");
  if (!f) return LACACHE_ERR_IO;
  FileHeader hdr;
  if (fread(&hdr, 1, sizeof hdr, f) != sizeof hdr || memcmp(hdr.magic, kFileMagic, sizeof kFileMagic) != 0 ||
      hdr.version != kFileVersion || hdr.header_bytes != sizeof hdr || hdr.n < 0) {
    fclose(f);
    return LACACHE_ERR_IO;
  }
  lacache_config cfg = hdr.cfg;
  cfg.device = device;
  if (capacity > 0) cfg.capacity = capacity;
  if (cfg.capacity < hdr.n) {
    fclose(f);
    return LACACHE_ERR_CAPACITY;
  }
  lacache_t* h = nullptr;
  lacache_status s = lacache_create_ensemble(&cfg, &hdr.ens, &h);
  if (s != LACACHE_OK) {
    fclose(f);
    return s;
  }
  DeviceGuard guard(h->cfg.device);
  const size_t n = (size_t)hdr.n;
  const size_t sizes[3] = {n * h->cfg.d * 2, n * h->pd * 2, n * h->cfg.k * 4};
  unsigned char* stage = nullptr;
  if (!guard.ok() || cudaMallocHost(&stage, kIoChunk) != cudaSuccess) {
    cudaGetLastError();
    s = LACACHE_ERR_OOM;
  } else if (!copy_in(f, h->key, sizes[0], stage) || !copy_in(f, h->prefix, sizes[1], stage) ||
             !copy_in(f, h->ids, sizes[2], stage)) {
    s = LACACHE_ERR_IO;
  }
  if (stage) cudaFreeHost(stage);
  fclose(f);
  if (s != LACACHE_OK) {
    lacache_destroy(h);
    return s;
  }
  h->n = hdr.n;
  *out = h;
  return LACACHE_OK;
}

lacache_status lacache_get_stats(lacache_t* h, lacache_stats* out, int32_t reset) {
  if (!h || !out) return LACACHE_ERR_INVALID_ARG;
  DeviceGuard guard(h->cfg.device);
  if (!guard.ok()) return LACACHE_ERR_CUDA;
  unsigned long long d[3];
  if (cudaDeviceSynchronize() != cudaSuccess ||
      cudaMemcpy(d, h->counters, sizeof d, cudaMemcpyDeviceToHost) != cudaSuccess)
    return LACACHE_ERR_CUDA;
  out->lookups = h->lookups;
  out->queries = h->queries;
  out->hits = (int64_t)d[0];
  out->rejects = (int64_t)d[1];
  out->key_misses = (int64_t)d[2];
  out->inserted = h->inserted;
  out->appended = h->appended;
  if (reset) {
    if (cudaMemset(h->counters, 0, sizeof d) != cudaSuccess) return LACACHE_ERR_CUDA;
    h->lookups = h->queries = h->inserted = h->appended = 0;
  }
  return LACACHE_OK;
}

lacache_status lacache_last_launch(const lacache_t* h, int32_t* n_splits, int32_t* stage1_kernel) {
  if (!h) return LACACHE_ERR_INVALID_ARG;
  if (n_splits) *n_splits = h->last_splits;
  if (stage1_kernel) *stage1_kernel = h->last_kernel;
  return LACACHE_OK;
}

}  // extern "C"
