// Sticky device error word and the slot-list validator.
//
// Kernels never trap: a unit whose slot id is out of range is skipped and the
// first such status is latched in a per-device word that stepq_device_error()
// reads and clears.
#include <atomic>

#include "device.cuh"
#include "internal.h"
#include "pipeline.cuh"

namespace stepq {

constexpr int kMaxDevices = 64;

__device__ unsigned int g_error_word;

// Device address of a file-scope __device__ variable on the current device,
// looked up once per device. The cache entries are atomics: host threads that
// make their first call on a device at the same time store the same address.
static void *symbol_address(const void *symbol, std::atomic<void *> (&cache)[kMaxDevices]) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    void *p = cache[dev].load(std::memory_order_acquire);
    if (!p) {
        if (cudaGetSymbolAddress(&p, symbol) != cudaSuccess || !p) return nullptr;
        cache[dev].store(p, std::memory_order_release);
    }
    return p;
}

unsigned int *device_error_word() {
    static std::atomic<void *> addr[kMaxDevices];
    return (unsigned int *)symbol_address((const void *)&g_error_word, addr);
}

// The pipelined kernels' wait bound and withheld item (test support). Plain
// process-wide values: stepq_debug_stall is documented as not thread-safe.
static long long g_wait_cycles = pipe::kWaitCycles;
static int g_withhold_item = -1;

StallKnob stall_knob() { return {g_wait_cycles, g_withhold_item}; }

stepq_status set_stall_knob(long long wait_cycles, int withhold_item) {
    if (wait_cycles < 1000 || withhold_item < -1) return STEPQ_ERR_ARG;
    g_wait_cycles = wait_cycles;
    g_withhold_item = withhold_item;
    return STEPQ_OK;
}

stepq_status read_device_error(cudaStream_t s) {
    unsigned int *w = device_error_word();
    if (!w) return STEPQ_ERR_CUDA;
    unsigned int v = 0;
    if (cudaMemcpyAsync(&v, w, sizeof(v), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaMemsetAsync(w, 0, sizeof(v), s) != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess)
        return STEPQ_ERR_CUDA;
    return (stepq_status)v;
}

// Marks each slot in a bitmap with atomicOr; a bit already set means a repeat.
__global__ void validate_slots_kernel(const int32_t *slots, int B, int pool_slots,
                                      uint32_t *bitmap, int32_t *status) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= B) return;
    const int s = slots[t];
    if (s < 0 || s >= pool_slots) {
        atomicCAS((unsigned int *)status, 0u, (unsigned int)STEPQ_ERR_SLOT_RANGE);
        return;
    }
    const uint32_t bit = 1u << (s & 31);
    if (atomicOr(&bitmap[s >> 5], bit) & bit)
        atomicCAS((unsigned int *)status, 0u, (unsigned int)STEPQ_ERR_DUP_SLOT);
}

stepq_status launch_validate_slots(const int32_t *slots, int B, int pool_slots,
                                   uint32_t *scratch, int32_t *status, cudaStream_t s) {
    if (cudaMemsetAsync(scratch, 0, ((size_t)pool_slots + 31) / 32 * 4, s) != cudaSuccess ||
        cudaMemsetAsync(status, 0, sizeof(int32_t), s) != cudaSuccess)
        return STEPQ_ERR_CUDA;
    if (B > 0) validate_slots_kernel<<<(B + 255) / 256, 256, 0, s>>>(slots, B, pool_slots, scratch, status);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

// ---- slot validation without allocation ----
// For callers that cannot allocate device memory and have no spare scratch to
// pass: the bitmap lives in this file-scope array, which every GPU that loads
// the library keeps for the life of the process.
constexpr int kStaticSlotMax = 1 << 20;                       // pool slots covered (128 KiB)
static __device__ __align__(256) uint32_t g_slot_bitmap[kStaticSlotMax / 32];

// Device address of the array on the current device, looked up once per device.
// Host code must not hand the symbol itself to a kernel: on the host it only
// names a stand-in, not device memory.
static uint32_t *static_bitmap(stepq_status *st) {
    static std::atomic<void *> addr[kMaxDevices];
    auto *p = (uint32_t *)symbol_address((const void *)g_slot_bitmap, addr);
    if (!p) *st = STEPQ_ERR_CUDA;
    return p;
}

stepq_status launch_validate_slots_static(const int32_t *slots, int B, int pool_slots,
                                          int32_t *status, cudaStream_t s) {
    if (pool_slots > kStaticSlotMax) return STEPQ_ERR_UNSUPPORTED;
    stepq_status st = STEPQ_OK;
    uint32_t *bitmap = static_bitmap(&st);
    if (!bitmap) return st;
    // the same validator; it clears the (pool_slots + 31) / 32 words it uses first
    return launch_validate_slots(slots, B, pool_slots, bitmap, status, s);
}

}  // namespace stepq
