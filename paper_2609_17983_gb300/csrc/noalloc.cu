// noalloc.cu -- kvr_linear_noalloc: a projection through the tensor-core GEMM
// that allocates nothing during the call.
//
// Who needs it: callers that must not allocate device memory at call time.
// Examples are a serving loop running under a fixed memory budget that was
// reserved up front, code that cannot afford the device-wide synchronisation
// cudaMalloc/cudaFree may imply, and hosts whose allocator is owned by
// someone else (a framework's pool it cannot call into).  Such callers own the
// input and output buffers themselves.  The GEMM's own scratch (the fp32
// partial tiles of split tiles and their arrival counters) therefore lives in
// the fixed device array below, reserved once when the library is loaded.
//
// Limits: at most NOALLOC_MAX_ROWS activation rows (one token tile of at most
// 64 rows) and at most NOALLOC_MAX_CTAS CTAs, so the partial tiles fit in
// NOALLOC_PARTIAL_FLOATS floats; at most NOALLOC_COUNTERS output tiles.  The
// array is ~10.5 MB of device memory that every GPU which loads the library
// keeps until the process exits.
//
// Pointers: x and y must be device (or managed) memory of the model's device;
// anything else is refused before the launch (a host address would reach the
// TMA descriptor and the epilogue stores).
//
// Lifetime: the array's device address is looked up once per device and kept
// until the process exits.  After cudaDeviceReset, or a release of the
// device's primary context, that address is stale: do not call this entry
// point on that device again in the same process.
//
// Sharing: every call uses the same array and leaves its contents behind.
// The arrival counters are cleared at the start of each call (stream-ordered
// memset, no allocation).  Calls whose GPU work overlaps in time (different
// streams, or different host threads on one device) race on the array and
// produce wrong results; serialise them on one stream.
#include <mutex>

#include "kvr_internal.cuh"

namespace {

constexpr int NOALLOC_MAX_ROWS = 64;
constexpr int NOALLOC_MAX_CTAS = 160;
constexpr int NOALLOC_COUNTERS = 8192;
constexpr size_t NOALLOC_PARTIAL_FLOATS = (size_t)NOALLOC_MAX_CTAS * 2 * NOALLOC_MAX_ROWS * 128;
constexpr size_t NOALLOC_PARTIAL_BYTES = NOALLOC_PARTIAL_FLOATS * sizeof(float);
constexpr size_t NOALLOC_COUNTER_BYTES = NOALLOC_COUNTERS * sizeof(int);
constexpr size_t NOALLOC_BYTES = NOALLOC_PARTIAL_BYTES + NOALLOC_COUNTER_BYTES;

// The scratch: [partials | counters].  In host code this name is only a
// host-side stand-in; kernels must be given the device address obtained with
// cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_BYTES];

constexpr int MAX_DEVICES = 64;
std::mutex g_mu;
void *g_scratch_dev[MAX_DEVICES] = {};

kvr_status na_fail(kvr_status code, const char *msg) {
  kvr::set_last_error(msg);  // reported by kvr_last_error()
  return code;
}

// Device address of the scratch on the current device (set-up once per
// device, with that device current).
kvr_status scratch_address(int device, void **out) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (device < 0 || device >= MAX_DEVICES) return na_fail(KVR_E_UNSUPPORTED, "device index");
  if (!g_scratch_dev[device]) {
    void *p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return na_fail(KVR_E_CUDA, cudaGetErrorString(e));
    g_scratch_dev[device] = p;
  }
  *out = g_scratch_dev[device];
  return KVR_OK;
}

// True if p is device or managed memory that `device` can use as such (the
// attribute query allocates nothing).
bool on_device(const void *p, int device) {
  cudaPointerAttributes a{};
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  if (a.type == cudaMemoryTypeManaged) return true;
  return a.type == cudaMemoryTypeDevice && a.device == device;
}

}  // namespace

using namespace kvr;

extern "C" kvr_status kvr_linear_noalloc(kvr_model *m, const char *name, int32_t layer,
                                         const void *x, int32_t M, float *y) {
  if (!m || !name || !x || !y) return na_fail(KVR_E_INVAL, "kvr_linear_noalloc: NULL argument");
  const Dims &dm = m->dims;
  if (dm.dtype != KVR_DTYPE_BF16 || !m->use_tc)
    return na_fail(KVR_E_UNSUPPORTED, "kvr_linear_noalloc: needs a bf16 model on the "
                                      "tensor-core GEMM");
  if (M < 1 || M > NOALLOC_MAX_ROWS)
    return na_fail(KVR_E_UNSUPPORTED,
                   "kvr_linear_noalloc: M must be in [1, 64] (the fixed scratch holds one "
                   "token tile of at most 64 rows)");
  std::string nm(name);
  const bool per_layer = nm != "lm_head";
  if (per_layer && (layer < 0 || layer >= dm.L))
    return na_fail(KVR_E_RANGE, "kvr_linear_noalloc: layer out of range");
  const LayerW *w = per_layer ? &m->layers[layer] : nullptr;
  const void *W = nullptr;
  const CUtensorMap *tm = nullptr;
  const float *bias = nullptr;
  int N = 0, K = 0;
  if (nm == "wqkv") {
    W = w->wqkv, tm = w->tc_qkv ? &w->tm_qkv : nullptr, bias = w->bqkv, N = dm.Nqkv(), K = dm.d;
  } else if (nm == "wo") {
    W = w->wo, tm = w->tc_o ? &w->tm_o : nullptr, N = dm.d, K = dm.H * dm.dh;
  } else if (nm == "wd") {
    W = w->wd, tm = w->tc_d ? &w->tm_d : nullptr, N = dm.d, K = dm.F;
  } else if (nm == "lm_head") {
    W = m->lm_head, tm = m->tc_lm ? &m->tm_lm : nullptr, N = dm.V, K = dm.d;
  } else {
    return na_fail(KVR_E_INVAL,
                   "kvr_linear_noalloc: name must be wqkv, wo, wd or lm_head");
  }
  if (!tm) return na_fail(KVR_E_UNSUPPORTED, "kvr_linear_noalloc: shape not on tensor cores");
  if ((long long)(N / 128) > NOALLOC_COUNTERS / 2)
    return na_fail(KVR_E_UNSUPPORTED, "kvr_linear_noalloc: more output tiles than counters");
  if (cudaSetDevice(m->device) != cudaSuccess)
    return na_fail(KVR_E_CUDA, "kvr_linear_noalloc: cudaSetDevice");
  if (!on_device(x, m->device) || !on_device(y, m->device))
    return na_fail(KVR_E_INVAL, "kvr_linear_noalloc: x and y must be device memory of the "
                                "model's device");
  void *scratch = nullptr;
  kvr_status st = scratch_address(m->device, &scratch);
  if (st) return st;
  TcWorkspace ws{};
  ws.partials = (float *)scratch;
  ws.counters = (int *)((unsigned char *)scratch + NOALLOC_PARTIAL_BYTES);
  ws.dev_flag = m->dev_flag;  // reported by kvr_synchronize
  ws.num_sms = m->num_sms < NOALLOC_MAX_CTAS ? m->num_sms : NOALLOC_MAX_CTAS;
  ws.max_tiles = NOALLOC_COUNTERS / 2;  // arrivals, then published parts
  // the counters must start at zero: clear whatever an earlier call left
  if (cudaMemsetAsync(ws.counters, 0, NOALLOC_COUNTER_BYTES, m->stream) != cudaSuccess)
    return na_fail(KVR_E_CUDA, "kvr_linear_noalloc: counter clear");
  GemmArgs g{x, W, bias, y, M, N, K, K, N, dm.dtype, 0};
  const char *e = launch_gemm_tc(g, *tm, GEMM_EPI_STORE, nullptr, 0, ws, m->stream);
  if (e) return na_fail(KVR_E_CUDA, e);
  return KVR_OK;
}
