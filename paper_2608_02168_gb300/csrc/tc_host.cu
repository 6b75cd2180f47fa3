// Host side of the tensor-core kernels: tensor-map encoding through the driver entry point (no
// link against libcuda), and the library's device status word.
#include <cudaTypedefs.h>

#include <atomic>

#include "tc_util.cuh"

namespace hg {

// The device this process's library state belongs to (-1 until the first call binds it).
static std::atomic<int> g_bound_device{-1};

hg_status device_guard() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    (void)cudaGetLastError();
    return HG_OK;  // no usable device: the call's own CUDA calls report it
  }
  int bound = -1;
  if (g_bound_device.compare_exchange_strong(bound, dev) || bound == dev) return HG_OK;
  set_error("this library is bound to device %d (its one-time set-up ran there); device %d is current", bound, dev);
  return HG_ERR_UNSUPPORTED;
}

__device__ int g_device_status = 0;

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

hg_status make_tmap_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) {
    set_error("cuTensorMapEncodeTiled is not available from the driver");
    return HG_ERR_CUDA;
  }
  if (((uintptr_t)base & 15) || (cols * 2) % 16 || box_rows == 0 || box_rows > 256) {
    set_error("tensor map: base must be 16-byte aligned, rows 16-byte multiples, box rows in 1..256");
    return HG_ERR_INVALID_ARG;
  }
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled failed (%d) for a %llu x %llu array", (int)r, (unsigned long long)rows,
              (unsigned long long)cols);
    return HG_ERR_CUDA;
  }
  return HG_OK;
}

// Self-test of the bounded waits: thread 0 of one CTA waits `polls` times on an mbarrier that
// nothing arrives at (no copy, store or MMA is in flight) and records the give-up in the status
// word, as every tensor-core kernel does when one of its waits runs out.
__global__ void selftest_bounded_wait(uint32_t polls, int* status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    tc::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !tc::mbar_wait_n(&bar, 0, polls)) record_device_error(status, tc::kErrTimeout);
}

// Resolved once per process on the current device (the library drives one GPU per process).
int* device_status_ptr() {
  static int* addr = nullptr;
  if (!addr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_device_status) == cudaSuccess) addr = static_cast<int*>(p);
  }
  return addr;
}

}  // namespace hg

extern "C" hg_status hg_selftest_bounded_wait(uint32_t polls, hg_stream stream) {
  hg::clear_error();
  HG_TRY(hg::device_guard());
  HG_REQUIRE(polls >= 1 && polls <= (1u << 20), "polls must be in [1, 2^20]");
  int* status = hg::device_status_ptr();
  HG_REQUIRE(status != nullptr, "device status word unavailable");
  return hg::launch("selftest_bounded_wait", hg::selftest_bounded_wait, dim3(1), dim3(32), 0,
                    reinterpret_cast<cudaStream_t>(stream), polls, status);
}

extern "C" hg_status hg_bind_device(int32_t device) {
  hg::clear_error();
  HG_REQUIRE(device >= 0, "device must be >= 0");
  int bound = -1;
  if (hg::g_bound_device.compare_exchange_strong(bound, device) || bound == device) return HG_OK;
  hg::set_error("this library is already bound to device %d", bound);
  return HG_ERR_UNSUPPORTED;
}
