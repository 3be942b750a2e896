// lacache_lookup_noalloc: the two-stage lookup for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc at all: code running under an allocator that owns all device memory (a
// serving runtime's memory pool or a framework's caching allocator that must not be bypassed), code that must not
// synchronize the device (cudaMalloc/cudaFree can), and plug-ins loaded into a process whose memory budget is
// fixed up front. The regular entry points need a handle, and lacache_create allocates the store and the stage-1
// scratch. This entry point instead takes the cache rows as caller-owned device arrays and keeps the stage-1
// partial lists in a fixed, file-scope device array of this library. It allocates nothing.
//
// The scratch array is kNoAllocScratchBytes (8 MiB). Every GPU that loads the library holds it until the process
// exits, and every call on that GPU shares it.
#include <cuda.h>
#include <math.h>

#include <mutex>

#include "internal.cuh"

namespace {

constexpr size_t kNoAllocScratchBytes = (size_t)8 << 20;   // the stated maximum
constexpr size_t kStatusBytes = 256;                         // device status word, first 256 bytes
constexpr int kMaxDevices = 64;

// The scratch: [status word | partial candidate lists | partial-list records]. In host code this name is only a
// host-side stand-in; kernels receive the device address found by cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

struct DeviceSetup {
  bool ready;
  unsigned char* scratch;   // device address of g_noalloc_scratch on this device
  int num_sms;
  lc::EncodeTiledFn encode; // TMA descriptor encoder (nullptr if the driver does not provide it)
};

std::mutex g_setup_mutex;
DeviceSetup g_setup[kMaxDevices];

// One-time set-up for `dev`, which must be the current device: the device address of the scratch array, the SM
// count, and the TMA descriptor encoder. Every field is written and read under the lock, and the caller gets its
// own copy. Nothing here allocates.
lacache_status setup_device(int dev, DeviceSetup* out) {
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  DeviceSetup& s = g_setup[dev];
  if (!s.ready) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess) return LACACHE_ERR_CUDA;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return LACACHE_ERR_CUDA;
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      s.encode = reinterpret_cast<lc::EncodeTiledFn>(fn);
    else
      cudaGetLastError();
    s.scratch = static_cast<unsigned char*>(ptr);
    s.num_sms = sms;
    s.ready = true;
  }
  *out = s;
  return LACACHE_OK;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace

extern "C" lacache_status lacache_lookup_noalloc(const lacache_config* cfg, int64_t n, const void* key_dev,
                                                 const void* prefix_dev, const int32_t* ids_dev, int32_t B,
                                                 const void* q_emb_dev, const void* q_prefix_dev,
                                                 const int32_t* q_ids_dev, const lacache_result* out,
                                                 void* cuda_stream) {
  lc::NvtxRange nvtx("lacache_lookup_noalloc");
  if (!cfg || !out || n < 0 || B < 1) return LACACHE_ERR_INVALID_ARG;
  const lacache_config c = *cfg;
  if (c.d <= 0 || c.k <= 0 || c.top_c <= 0 || isnan(c.tau_c) || isnan(c.tau_a)) return LACACHE_ERR_INVALID_ARG;
  if (c.check_mode < LACACHE_CHECK_EMB || c.check_mode > LACACHE_CHECK_BOTH) return LACACHE_ERR_INVALID_ARG;
  if (c.stage1 < LACACHE_STAGE1_AUTO || c.stage1 > LACACHE_STAGE1_STREAM) return LACACHE_ERR_INVALID_ARG;
  if (c.token_match_min > c.k) return LACACHE_ERR_INVALID_ARG;
  if (c.d % 8 != 0 || c.d > lc::kMaxD || c.k > lc::kMaxK || c.top_c > lc::kMaxTopC) return LACACHE_ERR_UNSUPPORTED;
  if (n > (int64_t)INT32_MAX) return LACACHE_ERR_UNSUPPORTED;
  if (!q_emb_dev || !q_prefix_dev || !q_ids_dev || !aligned16(q_emb_dev) || !aligned16(q_prefix_dev))
    return LACACHE_ERR_INVALID_ARG;
  if (n > 0 && (!key_dev || !prefix_dev || !ids_dev || !aligned16(key_dev) || !aligned16(prefix_dev)))
    return LACACHE_ERR_INVALID_ARG;
  if (!out->entry_id || !out->status || !out->key_score || !out->prefix_score || !out->token_matches ||
      !out->n_cand)
    return LACACHE_ERR_INVALID_ARG;
  // The batch must fit the fixed scratch with at least one partial list per query.
  const size_t per_split = (size_t)B * ((size_t)8 * c.top_c + sizeof(lc::PartMeta));
  const size_t room = kNoAllocScratchBytes - kStatusBytes - 256;
  if (per_split > room) return LACACHE_ERR_UNSUPPORTED;

  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess) return LACACHE_ERR_CUDA;
  if (c.device < 0 || c.device >= ndev || c.device >= kMaxDevices) return LACACHE_ERR_INVALID_ARG;
  int prev = 0;
  if (cudaGetDevice(&prev) != cudaSuccess) return LACACHE_ERR_CUDA;
  if (prev != c.device && cudaSetDevice(c.device) != cudaSuccess) return LACACHE_ERR_CUDA;

  lacache_status result = LACACHE_OK;
  DeviceSetup s;
  result = setup_device(c.device, &s);
  if (result == LACACHE_OK) {
    cudaStream_t st = (cudaStream_t)cuda_stream;
    int max_splits = (int)(room / per_split);
    if (max_splits > s.num_sms) max_splits = s.num_sms;
    unsigned int* status = reinterpret_cast<unsigned int*>(s.scratch);
    uint64_t* part_cand = reinterpret_cast<uint64_t*>(s.scratch + kStatusBytes);
    const size_t cand_bytes = ((size_t)max_splits * B * c.top_c * 8 + 255) & ~(size_t)255;
    lc::PartMeta* part_meta = reinterpret_cast<lc::PartMeta*>(s.scratch + kStatusBytes + cand_bytes);
    // Only the status word must start at zero; the stage-1 kernels write every partial entry they later read.
    if (cudaMemsetAsync(status, 0, sizeof(unsigned int), st) != cudaSuccess) result = LACACHE_ERR_CUDA;

    int splits = 0;
    if (result == LACACHE_OK && n > 0) {
      lc::Stage1Args a{};
      a.keys = reinterpret_cast<const __nv_bfloat16*>(key_dev);
      a.n = n;
      a.d = c.d;
      a.q = reinterpret_cast<const __nv_bfloat16*>(q_emb_dev);
      a.B = B;
      a.tau_c = c.tau_c;
      a.top_c = c.top_c;
      a.part_cand = part_cand;
      a.part_meta = part_meta;
      a.dev_status = status;
      // AUTO chooses as for a handle, and takes the streaming CUDA-core scan where the driver gives no TMA descriptor
      // encoder; an explicit TENSOR request without the encoder is an error
      int kernel = c.stage1 == LACACHE_STAGE1_AUTO ? lc::auto_stage1(n, c.d, B) : c.stage1;
      if (c.stage1 == LACACHE_STAGE1_AUTO && !s.encode) kernel = LACACHE_STAGE1_STREAM;
      cudaError_t e;
      if (kernel == LACACHE_STAGE1_TENSOR) {
        e = s.encode ? lc::launch_stage1_tensor(a, s.encode, s.num_sms, max_splits, st, &splits)
                     : cudaErrorInvalidValue;
      } else {
        e = lc::launch_stage1_stream(a, s.num_sms, max_splits, st, &splits);
      }
      if (e != cudaSuccess) result = LACACHE_ERR_CUDA;
    }
    if (result == LACACHE_OK) {
      lc::Stage2Args b{};
      b.n = n;
      b.part_cand = part_cand;
      b.part_meta = part_meta;
      b.splits = splits;
      b.B = B;
      b.pd = c.d;
      b.k = c.k;
      b.top_c = c.top_c;
      b.m = 1;
      b.seg[1] = c.d;
      b.tau_m[0] = c.tau_a;
      b.check_mode = c.check_mode;
      b.token_match_min = c.token_match_min;
      b.prefix = reinterpret_cast<const __nv_bfloat16*>(prefix_dev);
      b.ids = ids_dev;
      b.q_prefix = reinterpret_cast<const __nv_bfloat16*>(q_prefix_dev);
      b.q_ids = q_ids_dev;
      b.out = *out;
      if (lc::launch_stage2(b, st) != cudaSuccess) result = LACACHE_ERR_CUDA;
    }
  }
  if (prev != c.device) cudaSetDevice(prev);
  return result;
}
