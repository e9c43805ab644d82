// msf_unpatchify_noalloc: the de-embedding + unpatchify of one window
// position, with its scratch in a fixed device array instead of the plan's
// workspace, for callers that cannot allocate device memory.
//
// Some hosts never let a library allocate device memory: a serving runtime or
// plugin host that hands out every device buffer from its own pool and
// accounts for each byte, or a certified runtime that forbids allocation
// after start-up. cudaMalloc there would bypass the host's accounting, can
// synchronise the device, and fragments a pool the host manages. Such callers
// still need the emitted head state as a latent, so this entry point needs no
// workspace: the split-K fp32 partial sums and the raw token block live in
// g_noalloc_scratch, a file-scope __device__ array that every GPU which loads
// this library holds until the process exits.
#include <cuda_runtime.h>
#include <string.h>

#include <mutex>

#include "gemm_tc.h"
#include "internal.h"
#include "kernels.h"

namespace {

// Fixed scratch: [status word area | raw bf16 tokens [B][C*Hl*Wl] | fp32
// partial sums [splits][B][C*Hl*Wl]].
constexpr size_t kNoAllocScratchBytes = (size_t)8 << 20;  // 8 MiB
constexpr size_t kNoAllocStatusBytes = 256;
constexpr int kNoAllocMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mu;
void* g_noalloc_addr[kNoAllocMaxDevices];

// Device address of g_noalloc_scratch on the current device. In host code the
// symbol is only a stand-in, not a device address: kernels must be given the
// address looked up here, once per device, with that device current. The
// first lookup on a device also zeroes the status word at the start of the
// array (a synchronous cudaMemset, so it must not run under stream capture);
// after that only msf_noalloc_device_status clears it, so a timeout stays
// visible until it is read.
msf_status scratch_address(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        msf::set_cuda_error((int)e);
        return MSF_ERR_CUDA;
    }
    if (dev < 0 || dev >= kNoAllocMaxDevices) return MSF_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_addr[dev]) {
        void* ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
        if (e == cudaSuccess && !ptr) e = cudaErrorInvalidSymbol;
        if (e == cudaSuccess) e = cudaMemset(ptr, 0, kNoAllocStatusBytes);
        if (e != cudaSuccess) {
            msf::set_cuda_error((int)e);
            return MSF_ERR_CUDA;
        }
        g_noalloc_addr[dev] = ptr;
    }
    *out = g_noalloc_addr[dev];
    return MSF_OK;
}

}  // namespace

extern "C" msf_status msf_unpatchify_noalloc(msf_plan_t plan, int32_t position, const void* tokens,
                                             const void* w_out, void* latent_out, void* stream) {
    if (!plan || !tokens || !w_out || !latent_out) return MSF_ERR_INVALID_ARG;
    const msf::Plan& p = *plan;
    if (p.elem != 2 || p.d.latent_channels <= 0 || p.d.patch <= 0 || p.d.embed_dim <= 0)
        return MSF_ERR_UNSUPPORTED;
    if (position < 0 || position >= p.T) return MSF_ERR_INVALID_ARG;
    if (((uintptr_t)tokens & 15) || ((uintptr_t)w_out & 15) || ((uintptr_t)latent_out & 15))
        return MSF_ERR_INVALID_ARG;

    msf::MspShape sh;
    memset(&sh, 0, sizeof(sh));
    sh.T = p.T;
    sh.C = p.d.latent_channels;
    sh.patch = p.d.patch;
    sh.Hl = p.gh * p.d.patch;  // F latent frames stacked: [C, F, Hl, Wl] = [C, F*Hl, Wl]
    sh.Wl = p.d.grid_w * p.d.patch;
    for (int l = 0; l < p.T; ++l) sh.scales[l] = p.d.scales[l];
    const size_t per = (size_t)sh.C * sh.Hl * sh.Wl;  // elements per stream and state
    const size_t raw_bytes = msf::round256((size_t)p.B * per * 2);
    const size_t split_bytes = (size_t)p.B * per * 4;
    // Reject problems beyond the fixed scratch.
    if (kNoAllocStatusBytes + raw_bytes > kNoAllocScratchBytes) return MSF_ERR_UNSUPPORTED;
    const size_t room = kNoAllocScratchBytes - kNoAllocStatusBytes - raw_bytes;
    int max_splits = (int)(room / split_bytes);
    if (max_splits > msf::kMaxDeembedSplits) max_splits = msf::kMaxDeembedSplits;
    if (max_splits < 2) max_splits = 1;

    void* base = nullptr;
    msf_status st = scratch_address(&base);
    if (st != MSF_OK) return st;
    unsigned int* status = (unsigned int*)base;
    char* raw = (char*)base + kNoAllocStatusBytes;
    float* part = (float*)(raw + raw_bytes);
    cudaStream_t s = (cudaStream_t)stream;

    // The partial sums and raw tokens are fully overwritten by every call;
    // the status word keeps a timeout until msf_noalloc_device_status reads it.
    cudaError_t e;
    const int P = p.d.patch * p.d.scales[position];
    const int F = sh.C * P * P;
    const int E = p.d.embed_dim;
    msf::GemmTcArgs t;
    t.A = (const char*)tokens + (size_t)p.st_off[position] * E * 2;
    t.B = w_out;
    t.C = raw;
    t.M = p.st_n[position];
    t.N = F;
    t.K = E;
    t.lda = E;
    t.ldb = E;
    t.ldc = F;
    t.a_bstride = (long long)p.N * E;
    t.c_bstride = (long long)per;
    t.status = status;
    t.C32 = max_splits > 1 ? part : nullptr;
    t.max_splits = max_splits;
    if (!msf::gemm_tc_supported(t)) return MSF_ERR_UNSUPPORTED;
    e = msf::launch_gemm_tc(t, p.B, s);
    if (e == cudaSuccess) {
        if (t.splits_used > 1)
            e = msf::launch_unpatchify_splitk(part, t.splits_used, latent_out, sh, position, p.B, s);
        else
            e = msf::launch_unpatchify_raw(raw, latent_out, sh, position, (long long)per, 0, p.B,
                                           true, s);
    }
    if (e != cudaSuccess) {
        msf::set_cuda_error((int)e);
        return MSF_ERR_CUDA;
    }
    return MSF_OK;
}

extern "C" msf_status msf_noalloc_device_status(void* stream) {
    void* base = nullptr;
    msf_status st = scratch_address(&base);
    if (st != MSF_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    unsigned int word = 0;
    cudaError_t e = cudaStreamSynchronize(s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&word, base, sizeof(word), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(base, 0, sizeof(word), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) {
        msf::set_cuda_error((int)e);
        return MSF_ERR_CUDA;
    }
    return word ? MSF_ERR_TIMEOUT : MSF_OK;
}

extern "C" msf_status msf_noalloc_selftest_wait_timeout(int64_t limit_cycles, void* stream) {
    if (limit_cycles < 1 || limit_cycles > (int64_t(1) << 31)) return MSF_ERR_INVALID_ARG;
    void* base = nullptr;
    msf_status st = scratch_address(&base);
    if (st != MSF_OK) return st;
    cudaError_t e = msf::launch_wait_timeout_selftest((unsigned int*)base, (long long)limit_cycles,
                                                      (cudaStream_t)stream);
    if (e != cudaSuccess) {
        msf::set_cuda_error((int)e);
        return MSF_ERR_CUDA;
    }
    return MSF_OK;
}
