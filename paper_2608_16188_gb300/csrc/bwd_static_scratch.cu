// bwd_static_scratch.cu -- vmoe_expert_bwd for callers that cannot allocate
// device memory.
//
// vmoe_expert_bwd needs a dH buffer that the caller allocates and passes in.
// Some callers cannot do that: a plug-in whose host framework owns every
// device buffer and hands out only its own tensors, or a deployment that
// forbids any device allocation after start-up (fixed memory budgets that are
// certified once).  This entry point gives them the same backward with its
// scratch in a fixed array that lives in the library itself.
//
// When dH for every group does not fit, the bf16 backward runs in slices of
// groups planned to fit the array (vmoe_expert_bwd with a smaller workspace),
// which reads the loads back to the host and synchronises the stream.  Only a
// problem whose smallest workspace (one group's dH, or all of an fp32
// problem's dH) exceeds the array is refused.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds VMOE_STATIC_SCRATCH_BYTES of it until the process exits.  In
// host code its name is only a host-side stand-in, so the device address is
// looked up once per device with cudaGetSymbolAddress (with that device
// current) and cached; kernels receive that address like any workspace.
#include "common.cuh"

namespace {

static __device__ __align__(256) unsigned char g_bwd_scratch[VMOE_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
// Per-device cache of the array's device address.  Host threads may call
// concurrently; each stores the same value, published with release order.
std::atomic<void *> g_scratch_addr[kMaxDevices];

}  // namespace

extern "C" int vmoe_expert_bwd_static_scratch(const vmoe_problem *p, const void *xe, const void *h,
                                              const void *a, const void *w1, const void *w2,
                                              const void *dye, const int32_t *load, void *dxe,
                                              void *dw1, void *dw2, void *cuda_stream) {
    // dH for every group, or -- bf16 -- at least one group's, which runs the
    // backward in slices planned to fit the array
    const size_t need = vmoe_expert_bwd_min_workspace_size(p);
    if (need == 0) return VMOE_ERR_INVALID;                       // invalid problem statement
    if (need > VMOE_STATIC_SCRATCH_BYTES) return VMOE_ERR_UNSUPPORTED;  // too large for the array
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return VMOE_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return VMOE_ERR_UNSUPPORTED;
    void *addr = g_scratch_addr[dev].load(std::memory_order_acquire);
    if (addr == nullptr) {  // first call on this device: resolve the address
        if (cudaGetSymbolAddress(&addr, g_bwd_scratch) != cudaSuccess || addr == nullptr)
            return VMOE_ERR_CUDA;
        g_scratch_addr[dev].store(addr, std::memory_order_release);
    }
    // dH needs no clearing: the backward writes every row it later reads.
    return vmoe_expert_bwd(p, xe, h, a, w1, w2, dye, load, dxe, dw1, dw2, addr,
                           VMOE_STATIC_SCRATCH_BYTES, cuda_stream);
}
