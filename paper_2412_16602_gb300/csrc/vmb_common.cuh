// vmb_common.cuh - device helpers shared by the sm_103a kernels of libvmb:
// storage-type conversion, the fp32 fast math of the discretisation, and the
// bounded decoupled look-back used to carry the scan state across L-chunks.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace vmb {

constexpr float kLog2e = 1.4426950408889634f;

// ------------------------------------------------------------ storage types

template <typename T> struct io;
template <> struct io<float> {
    static __device__ __forceinline__ float ld(const float* p) { return *p; }
    static __device__ __forceinline__ float cvt(float v) { return v; }
    static __device__ __forceinline__ float to(float v) { return v; }
};
template <> struct io<__nv_bfloat16> {
    static __device__ __forceinline__ float ld(const __nv_bfloat16* p) { return __bfloat162float(*p); }
    static __device__ __forceinline__ float cvt(__nv_bfloat16 v) { return __bfloat162float(v); }
    // round to nearest even
    static __device__ __forceinline__ __nv_bfloat16 to(float v) { return __float2bfloat16_rn(v); }
};

// ------------------------------------------------------------------- math

// 2^x on the MUFU pipe (ex2.approx, flush-to-zero).  Relative error about
// 2^-22 over the range the scan uses; the parity tests bound its effect.
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float rcp(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// softplus(v) = log(1 + e^v) (Eq. 6, tau_Delta), written as
// max(v, 0) + log1p(e^-|v|).  log1p(e) for e in (0, 1] uses the series
// log1p(e) = 2 atanh(z) = 2 z (1 + z^2/3 + z^4/5 + ...), z = e / (2 + e) <= 1/3
// (Abramowitz & Stegun 4.1.27), truncated after z^12/13: truncation error below
// (1/3)^14 / 15 ~ 1.4e-8 relative, so the result keeps the relative accuracy of
// e^-|v| even where log1p(e) is tiny.  No cut-off for large |v|.
__device__ __forceinline__ float softplus_from_e(float v, float e) {
    float z = e * rcp(2.0f + e);
    float w = z * z;
    float p = 1.0f / 13.0f;
    p = fmaf(p, w, 1.0f / 11.0f);
    p = fmaf(p, w, 1.0f / 9.0f);
    p = fmaf(p, w, 1.0f / 7.0f);
    p = fmaf(p, w, 1.0f / 5.0f);
    p = fmaf(p, w, 1.0f / 3.0f);
    p = fmaf(p, w, 1.0f);
    return fmaxf(v, 0.0f) + 2.0f * z * p;
}
// e = e^-|v| (ex2.approx), shared with the derivative below
__device__ __forceinline__ float softplus_e(float v) { return ex2(-fabsf(v) * kLog2e); }
__device__ __forceinline__ float softplus(float v) { return softplus_from_e(v, softplus_e(v)); }

// softplus'(v) = the logistic function 1 / (1 + e^-v), from e = e^-|v| (no
// overflow): 1 / (1 + e) for v >= 0, e / (1 + e) otherwise.
__device__ __forceinline__ float softplus_grad_from_e(float v, float e) {
    const float r = rcp(1.0f + e);
    return v >= 0.0f ? r : e * r;
}

// softplus of two values with the packed f32x2 operations (the same operations
// as softplus() applied to each value, issued as one instruction per pair
// where the FMA pipe allows it); softplus2_from_e takes e = e^-|v| of both.
__device__ __forceinline__ float2 softplus2_e(float2 v) {
    const float2 av = make_float2(__int_as_float(__float_as_int(v.x) & 0x7fffffff),
                                  __int_as_float(__float_as_int(v.y) & 0x7fffffff));
    const float2 m = __fmul2_rn(av, make_float2(-kLog2e, -kLog2e));
    return make_float2(ex2(m.x), ex2(m.y));
}
__device__ __forceinline__ float2 softplus2_from_e(float2 v, float2 e) {
    const float2 den = __fadd2_rn(e, make_float2(2.0f, 2.0f));
    const float2 z = __fmul2_rn(e, make_float2(rcp(den.x), rcp(den.y)));
    const float2 w = __fmul2_rn(z, z);
    float2 q = make_float2(1.0f / 13.0f, 1.0f / 13.0f);
    q = __ffma2_rn(q, w, make_float2(1.0f / 11.0f, 1.0f / 11.0f));
    q = __ffma2_rn(q, w, make_float2(1.0f / 9.0f, 1.0f / 9.0f));
    q = __ffma2_rn(q, w, make_float2(1.0f / 7.0f, 1.0f / 7.0f));
    q = __ffma2_rn(q, w, make_float2(1.0f / 5.0f, 1.0f / 5.0f));
    q = __ffma2_rn(q, w, make_float2(1.0f / 3.0f, 1.0f / 3.0f));
    q = __ffma2_rn(q, w, make_float2(1.0f, 1.0f));
    const float2 z2 = __fadd2_rn(z, z);
    return __ffma2_rn(z2, q, make_float2(fmaxf(v.x, 0.0f), fmaxf(v.y, 0.0f)));
}
__device__ __forceinline__ float2 softplus2(float2 v) { return softplus2_from_e(v, softplus2_e(v)); }

// ------------------------------------------- programmatic dependent launch

// Every kernel of libvmb is launched with programmatic stream serialization,
// so that its CTAs can be scheduled while the previous kernel of the stream
// drains.  Each kernel therefore executes pdl_wait() (griddepcontrol.wait:
// the previous kernel has completed and its writes are visible) before it
// touches global memory, and only then pdl_launch_dependents(), which lets
// the next kernel be scheduled.  Because no kernel signals its dependents
// before its own wait has returned, a kernel that is already running may
// read data written two or more launches earlier before its own wait (the
// third launch of the chunked full scan does so).  Both instructions are
// no-ops in a kernel launched without the attribute.
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Host side: launch `fn` with the programmatic attribute set.
// programmatic = false: an ordinary launch (the kernel starts after the
// previous one has completed; its pdl_wait returns at once).  Used for grids
// of long-lived CTAs: launched early, they are placed on the SMs that the
// previous kernel frees first, up to the per-SM limit, and leave the others
// idle for their whole life.
inline cudaError_t launch_kernel(const void* fn, dim3 grid, dim3 block, size_t smem, void** args,
                                 cudaStream_t stream, bool programmatic = true) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = programmatic ? attr : nullptr;
    cfg.numAttrs = programmatic ? 1 : 0;
    return cudaLaunchKernelExC(&cfg, fn, args);
}

// ------------------------------------------------------ memory-model helpers

__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release(unsigned* p, unsigned v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned ld_relaxed(const unsigned* p) {
    unsigned v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ float ld_cg(const float* p) { return __ldcg(p); }
__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ------------------------------------------------------- workspace / look-back

// Status header at the start of every scan workspace (256 bytes).
struct WsHeader {
    unsigned ticket;     // next CTA ticket of the running launch
    unsigned done;       // CTAs of the running launch that have finished
    unsigned gen;        // launch generation: tags the chunk flags of one launch
    unsigned err;        // error bits (kErrTimeout, kErrBounds), cleared by vmb_read_status
    unsigned err_seq;    // first sequence / chunk whose wait gave up (diagnostics)
    unsigned err_chunk;
    unsigned pad[58];
};
static_assert(sizeof(WsHeader) == 256, "header is 256 bytes");

constexpr unsigned kErrTimeout = 1u;
constexpr unsigned kErrBounds = 2u;
constexpr unsigned kFlagAggregate = 1u;  // chunk aggregate published
constexpr unsigned kFlagInclusive = 2u;  // chunk inclusive prefix (end state) published
constexpr uint64_t kWaitLimitNs = 200ull * 1000ull * 1000ull;  // 0.2 s per wait

__device__ __forceinline__ unsigned flag_word(unsigned gen, unsigned kind) {
    return ((gen & 0x3FFFFFFFu) << 2) | kind;
}

// Warp-wide look-back (call from one full warp; every lane gets the result).
// Finds the nearest predecessor j < chunk whose inclusive state is published
// such that every chunk in (j, chunk) has at least its aggregate published;
// the lanes poll 32 predecessor flags per round.  Returns -1 when the wait ran
// out or another CTA already reported an error.
__device__ __forceinline__ int lookback_find(const unsigned* flags, int chunk, unsigned gen, WsHeader* hdr,
                                             unsigned seq) {
    const unsigned tag = gen & 0x3FFFFFFFu;
    const int lane = threadIdx.x & 31;
    int hi = chunk - 1;
    const uint64_t t0 = globaltimer_ns();
    unsigned ns = 32;
    for (unsigned it = 0;; ++it) {
        const int j = hi - lane;
        unsigned kind = 0;
        if (j >= 0) {
            const unsigned f = ld_acquire(&flags[j]);
            kind = ((f >> 2) == tag) ? (f & 3u) : 0u;
        }
        const unsigned inc = __ballot_sync(0xffffffffu, kind == kFlagInclusive);
        const unsigned valid = __ballot_sync(0xffffffffu, kind != 0 || j < 0);
        if (inc) {
            const int l = __ffs(inc) - 1;
            const unsigned need = l == 0 ? 0u : ((1u << l) - 1u);
            if ((valid & need) == need) return hi - l;
        } else if (valid == 0xffffffffu && hi >= 32) {
            hi -= 32;  // the whole window has aggregates: look further back
            continue;
        }
        if ((it & 15u) == 0) {
            unsigned stop = 0;
            if (lane == 0) {
                if (ld_relaxed(&hdr->err)) {
                    stop = 1;
                } else if (globaltimer_ns() - t0 > kWaitLimitNs) {
                    if (atomicOr(&hdr->err, kErrTimeout) == 0) {
                        hdr->err_seq = seq;
                        hdr->err_chunk = (unsigned)chunk;
                    }
                    stop = 1;
                }
            }
            if (__shfl_sync(0xffffffffu, stop, 0)) return -1;
        }
        __nanosleep(ns);
        if (ns < 1024) ns <<= 1;
    }
}

// Block-wide look-back: every thread of a CTA of NT threads calls it, thread i
// polls predecessor hi - i, so one round covers NT predecessors instead of 32.
// Same contract as lookback_find (returns the nearest predecessor whose
// inclusive state is published with every chunk after it at least aggregated,
// or -1 when the wait ran out or another CTA reported an error).  s_scr holds
// 2 NT / 32 + 2 words of shared memory.
template <int NT>
__device__ __forceinline__ int lookback_find_block(const unsigned* flags, int chunk, unsigned gen, WsHeader* hdr,
                                                   unsigned seq, unsigned* s_scr) {
    constexpr int NW = NT / 32;
    constexpr int kRetry = -2;
    const unsigned tag = gen & 0x3FFFFFFFu;
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    int hi = chunk - 1;
    const uint64_t t0 = globaltimer_ns();
    unsigned ns = 32;
    for (unsigned it = 0;; ++it) {
        const int j = hi - tid;
        unsigned kind = 0;
        if (j >= 0) {
            const unsigned f = ld_acquire(&flags[j]);
            kind = ((f >> 2) == tag) ? (f & 3u) : 0u;
        }
        const unsigned inc = __ballot_sync(0xffffffffu, kind == kFlagInclusive);
        const unsigned valid = __ballot_sync(0xffffffffu, kind != 0 || j < 0);
        if (lane == 0) {
            s_scr[w] = inc;
            s_scr[NW + w] = valid;
        }
        __syncthreads();
        if (tid == 0) {
            int res = kRetry, nhi = hi;
            bool decided = false;
            for (int ww = 0; ww < NW && !decided; ++ww) {
                const unsigned iv = s_scr[ww], vv = s_scr[NW + ww];
                if (iv) {
                    const int l = __ffs(iv) - 1;
                    const unsigned need = l == 0 ? 0u : ((1u << l) - 1u);
                    if ((vv & need) == need) res = hi - (ww * 32 + l);
                    decided = true;
                } else if (vv != 0xffffffffu) {
                    decided = true;  // a predecessor has published nothing yet
                }
            }
            if (!decided && hi >= NT) {
                nhi = hi - NT;  // the whole window is aggregated: look further back
                res = kRetry - 1;
            }
            if (res == kRetry && (it & 15u) == 0) {
                if (ld_relaxed(&hdr->err)) {
                    res = -1;
                } else if (globaltimer_ns() - t0 > kWaitLimitNs) {
                    if (atomicOr(&hdr->err, kErrTimeout) == 0) {
                        hdr->err_seq = seq;
                        hdr->err_chunk = (unsigned)chunk;
                    }
                    res = -1;
                }
            }
            s_scr[2 * NW] = (unsigned)res;
            s_scr[2 * NW + 1] = (unsigned)nhi;
        }
        __syncthreads();
        const int res = (int)s_scr[2 * NW];
        hi = (int)s_scr[2 * NW + 1];
        __syncthreads();  // s_scr is rewritten by the next round
        if (res >= -1) return res;
        if (res == kRetry) {
            __nanosleep(ns);
            if (ns < 1024) ns <<= 1;
        }
    }
}

// Called by thread 0 of every CTA of a look-back launch once the CTA is done
// with the workspace: the last CTA resets the ticket and completion counters
// and advances the generation, leaving the workspace ready for the next launch.
__device__ __forceinline__ void finish_launch(WsHeader* hdr, unsigned total_ctas) {
    __threadfence();
    unsigned prev = atomicAdd(&hdr->done, 1u);
    if (prev == total_ctas - 1) {
        __threadfence();
        hdr->ticket = 0;
        hdr->done = 0;
        atomicAdd(&hdr->gen, 1u);
        __threadfence();
    }
}

// ------------------------------------------------------ L2 eviction policies

// Cache policies for loads/stores with an L2 eviction hint (sm_80+ createpolicy):
// evict_last keeps data that is read again soon, evict_first streams data
// through without displacing it.
__device__ __forceinline__ uint64_t l2_evict_last() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t l2_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ float ld_hint(const float* p, uint64_t pol) {
    float v;
    asm volatile("ld.global.L2::cache_hint.f32 %0, [%1], %2;" : "=f"(v) : "l"(p), "l"(pol));
    return v;
}
__device__ __forceinline__ float ld_hint(const __nv_bfloat16* p, uint64_t pol) {
    unsigned short v;
    asm volatile("ld.global.L2::cache_hint.b16 %0, [%1], %2;" : "=h"(v) : "l"(p), "l"(pol));
    return __uint_as_float((unsigned)v << 16);
}
__device__ __forceinline__ void st_hint(float* p, float v, uint64_t pol) {
    asm volatile("st.global.L2::cache_hint.f32 [%0], %1, %2;" ::"l"(p), "f"(v), "l"(pol) : "memory");
}
__device__ __forceinline__ void st_hint(__nv_bfloat16* p, float v, uint64_t pol) {
    const unsigned short b = __bfloat16_as_ushort(__float2bfloat16_rn(v));
    asm volatile("st.global.L2::cache_hint.b16 [%0], %1, %2;" ::"l"(p), "h"(b), "l"(pol) : "memory");
}

// --------------------------------------------------------- async copies

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, int src_bytes) {
    unsigned s = (unsigned)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(s), "l"(gmem), "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// ------------------------------------------- mbarriers and tensor copies (TMA)

// Shared-memory mbarriers (one CTA; no cluster) and the tiled bulk tensor copy
// global -> shared that signals one of them with its byte count.
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbarrier_init(uint32_t bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbarrier_expect_tx(uint32_t bar, unsigned bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbarrier_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbarrier_test(uint32_t bar, uint32_t parity) {
    uint32_t done;
    asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
                 : "=r"(done)
                 : "r"(bar), "r"(parity)
                 : "memory");
    return done != 0;
}
// Wait for the phase with the given parity to complete, bounded by `limit_ns`
// of wall time (false: the wait gave up).
__device__ __forceinline__ bool mbarrier_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
    if (mbarrier_test(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
        if (mbarrier_test(bar, parity)) return true;
        if (globaltimer_ns() - t0 > limit_ns) return false;
    }
}
// Tiled 3-D tensor copy (innermost coordinate x first) into shared memory,
// completing `bar`'s transaction count with the box's bytes.  Elements of the
// box outside the tensor are zero-filled.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const void* tensor_map, int x, int y, int z, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tensor_map)), "r"(x), "r"(y), "r"(z), "r"(bar)
        : "memory");
}

}  // namespace vmb
