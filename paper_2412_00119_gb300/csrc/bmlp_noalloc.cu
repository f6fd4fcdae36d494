// bmlp_noalloc.cu -- forward-only evaluation that allocates no memory.
//
// bmlp_predict keeps its inter-layer activations in device buffers that it
// allocates with cudaMalloc the first time it needs them.  Some callers cannot
// allow that: code running inside a region that forbids allocation (a host
// callback, a real-time or safety loop with a fixed memory plan, a process
// whose allocator is owned by another runtime).  bmlp_predict_noalloc runs the
// same kernels with its scratch in the fixed, file-scope device array below, so
// it never calls cudaMalloc, cudaFree or any allocating library routine.
#include <mutex>

#include "bmlp_internal.cuh"

namespace {

// Two ping-pong activation buffers of kNoallocWords 64-bit words each (16 MiB
// in total).  Every GPU that loads the library holds this array until exit.
constexpr int64_t kNoallocWords = 1 << 20;
__device__ __align__(256) uint64_t g_noalloc_scratch[2 * kNoallocWords];

// Device address of g_noalloc_scratch, looked up once per device.
std::mutex g_noalloc_mutex;
uint64_t* g_noalloc_ptr[64] = {nullptr};

int noalloc_scratch(uint64_t** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    (void)cudaGetLastError();
    return BMLP_ECUDA;
  }
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
      (void)cudaGetLastError();
      return BMLP_ECUDA;
    }
    g_noalloc_ptr[dev] = static_cast<uint64_t*>(p);
  }
  *out = g_noalloc_ptr[dev];
  return BMLP_OK;
}

}  // namespace

// Defined in bmlp_api.cu: the model geometry this entry point needs.
int bmlp_internal_eval_view(const bmlp_t* h, const bk::StepParams** params, int* nwmax);
int bmlp_internal_fail(bmlp_t* h, int code, const char* msg);
void bmlp_internal_clear_error(bmlp_t* h);
void bmlp_internal_count_launches(bmlp_t* h, int64_t n);

extern "C" int bmlp_predict_noalloc(bmlp_t* h, const uint64_t* x_packed, int64_t n,
                                    int32_t* labels_out, void* cuda_stream) {
  const bk::StepParams* P = nullptr;
  int nwmax = 0;
  if (bmlp_internal_eval_view(h, &P, &nwmax) != BMLP_OK) return BMLP_EINVAL;
  bmlp_internal_clear_error(h);
  if (n < 0) return bmlp_internal_fail(h, BMLP_EINVAL, "n < 0");
  if (n == 0) return BMLP_OK;
  if (!x_packed || !labels_out) return bmlp_internal_fail(h, BMLP_EINVAL, "x or labels_out is NULL");
  // nwmax >= 1; the quotient form cannot overflow for any caller-supplied n
  if (n > kNoallocWords / nwmax)
    return bmlp_internal_fail(h, BMLP_EINVAL,
                              "n exceeds the fixed scratch: at most 1048576 / ceil(max K_l / 64) rows");
  int cur_dev = 0;
  if (cudaGetDevice(&cur_dev) != cudaSuccess) {
    (void)cudaGetLastError();
    return bmlp_internal_fail(h, BMLP_ECUDA, "cudaGetDevice failed");
  }
  cudaPointerAttributes a;
  for (const void* p : {static_cast<const void*>(x_packed), static_cast<const void*>(labels_out)}) {
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess ||
        !(a.type == cudaMemoryTypeManaged || (a.type == cudaMemoryTypeDevice && a.device == cur_dev))) {
      (void)cudaGetLastError();
      return bmlp_internal_fail(h, BMLP_EINVAL,
                                "x and labels_out must be device pointers on the current device");
    }
  }
  uint64_t* scratch = nullptr;
  if (noalloc_scratch(&scratch) != BMLP_OK)
    return bmlp_internal_fail(h, BMLP_ECUDA, "cudaGetSymbolAddress of the scratch array failed");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const uint64_t* in = x_packed;
  uint64_t* buf[2] = {scratch, scratch + kNoallocWords};
  int cur = 0;
  for (int l = 1; l <= P->L; ++l) {
    const bk::DevLayer& D = P->layer[l - 1];
    bk::k_forward_eval<<<bk::eval_forward_grid(n, D.Kout), bk::eval_forward_block(), 0, st>>>(
        in, n, D.nw_in, D.W, D.Kout, D.Kin, buf[cur], D.nw_out);
    in = buf[cur];
    cur ^= 1;
  }
  const bk::DevLayer& DL = P->layer[P->L - 1];
  bk::k_predict_out<<<(unsigned)((n + 7) / 8), 256, 0, st>>>(in, n, DL.nw_out, DL.PT, P->c,
                                                             DL.Kout, labels_out);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return bmlp_internal_fail(h, BMLP_ECUDA, cudaGetErrorString(e));
  bmlp_internal_count_launches(h, P->L + 1);
  return BMLP_OK;
}
