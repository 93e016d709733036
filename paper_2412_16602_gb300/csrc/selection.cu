// selection.cu - the selection functions of Eq. 6: B, C and the raw Delta of
// every step as linear maps of the scan input u (the D channels of one step of
// one direction), with per-direction weights:
//   Bs[b,k,n,l] = sum_d WB[k,n,d] u[b,k,d,l],   Cs[b,k,n,l] = sum_d WC[k,n,d] u[b,k,d,l]
//   z[r] = sum_d Wz[k,r,d] u[b,k,d,l],          delta_raw[b,k,d,l] = sum_r Wup[k,d,r] z[r]
// (the printed s_Delta = Broadcast_D(Linear_1(u)) is R = 1 with unit Wup).
//
// Per (b, k) this is one dense contraction, P = W u with W = [WB; WC; Wz]
// ([2N + R, D]) and u ([D, L]), followed by a rank-R expansion.  It runs on the
// fifth-generation tensor cores: a CTA of 128 threads owns 128 steps of one
// (b, k) (the MMA's M = 128 rows are steps, one TMEM lane each), the output
// columns are B (0..15), C (16..31) and z (32..47) (N = 48), and the D channels
// are the reduction dimension, staged 16 at a time (the next chunk's loads are
// in flight while the tensor cores work on the current one).  Operands are fp32 in the
// tensor cores' tf32 format; to keep fp32 accuracy each value is split into a
// tf32 head and a tf32 tail (x = hi + lo, both exact in fp32) and the product is
// accumulated as hi.hi + hi.lo + lo.hi in fp32 (the lo.lo term is below fp32
// resolution).  bf16 inputs are exact in tf32 and need no tail.  The
// accumulator lives in TMEM; each thread reads back its step's 48 values and
// writes B, C and the D raw Deltas (z expanded through Wup in registers).
#include <stdint.h>

#include <mutex>

#include "vmb_common.cuh"
#include "vmb_internal.h"

namespace vmb {
namespace {

constexpr int kSelThreads = 128;  // steps per CTA = MMA rows = TMEM lanes
constexpr int kSelKC = 16;        // channels per staged chunk (two MMA k-steps of 8)
constexpr int kSelCols = 48;      // MMA N: B at columns 0..15, C at 16..31, z at 32..47
constexpr int kSelTmemCols = 64;  // TMEM allocation (a power of two >= 32)
constexpr int kSelRP = 16;        // z values per step held in registers (R <= 16)
constexpr int kSelDB = 256;       // Wup rows staged at a time in the epilogue
constexpr int kSelDrain = 16;     // chunks (256 channels) accumulated in TMEM before a drain to registers

struct SelParams {
    const void* u;
    const float* WB;
    const float* WC;
    const float* Wz;
    const float* Wup;
    void* Bs;
    void* Cs;
    void* dr;
    float* z;  // not null: the rank-R intermediate z [B,K,R,L] fp32 is written instead of dr
    int K, D, N, R, L;
    int nlb;  // step blocks per (b, k)
};

// Shared memory: the two operands of one chunk in the tensor cores' K-major
// layout without swizzle.  A core matrix is 8 rows x 16 bytes (4 tf32) stored
// as 128 contiguous bytes; core matrix (row group g, channel quad c) of an
// operand with G row groups sits at ((c * G) + g) * 128 bytes, so the stride
// between row groups is 128 bytes and between channel quads G * 128 bytes.
struct SelLayout {
    static constexpr size_t a_bytes = (size_t)kSelThreads * kSelKC * 4;  // u^T rows (steps): 16 KB
    static constexpr size_t b_bytes = (size_t)kSelCols * kSelKC * 4;     // W rows (outputs): 6 KB
    static constexpr size_t a_hi = 0, a_lo = a_bytes, b_hi = 2 * a_bytes, b_lo = 2 * a_bytes + b_bytes;
    static constexpr size_t bytes = 2 * a_bytes + 2 * b_bytes;
    static_assert((size_t)kSelDB * kSelRP * 4 <= bytes, "the epilogue's Wup rows reuse the operand area");
};

__device__ __forceinline__ uint32_t smem_addr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

// Round to the nearest tf32 value (10 stored mantissa bits; the low 13 bits become zero).
__device__ __forceinline__ float to_tf32(float x) {
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return __uint_as_float(r);
}

// Shared-memory matrix descriptor of the tensor cores: start address, leading
// (channel-quad) and stride (row-group) byte offsets, all in 16-byte units,
// descriptor version 1, no swizzle.
__device__ __forceinline__ uint64_t mma_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr >> 4) & 0x3FFF) | ((uint64_t)((lbo >> 4) & 0x3FFF) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFF) << 32) | ((uint64_t)1 << 46);
}

// Instruction descriptor of kind::tf32: fp32 accumulator, tf32 A and B, both
// K-major, N = kSelCols, M = kSelThreads.
constexpr uint32_t kSelIdesc = (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(kSelCols >> 3) << 17) |
                               ((uint32_t)(kSelThreads >> 4) << 24);

__device__ __forceinline__ void mma_tf32(uint32_t tmem, uint64_t da, uint64_t db, uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem),
        "l"(da), "l"(db), "r"(kSelIdesc), "r"(accumulate));
}

// Wait (bounded by 1 s of wall time) for the given phase of an mbarrier.
__device__ __forceinline__ bool mbar_wait(uint32_t mbar, uint32_t phase) {
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
        uint32_t done;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
            : "=r"(done)
            : "r"(mbar), "r"(phase)
            : "memory");
        if (done) return true;
        if (globaltimer_ns() - t0 > 1000000000ull) return false;
    }
}

template <typename T>
__global__ void __launch_bounds__(kSelThreads, 5) selection_kernel(const SelParams p) {
    using LY = SelLayout;
    constexpr bool F32 = sizeof(T) == 4;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint32_t s_tmem;
    __shared__ __align__(8) uint64_t s_mbar;
    pdl_wait();
    pdl_launch_dependents();
    const int tid = threadIdx.x, warp = tid / 32;
    const long long bk = blockIdx.x / p.nlb;
    const int k = (int)(bk % p.K);
    const int l = (int)(blockIdx.x % p.nlb) * kSelThreads + tid;
    const bool lv = l < p.L;
    const int D = p.D, N = p.N, R = p.R, L = p.L;

    // TMEM accumulator (warp 0 allocates) and the MMA-completion barrier
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&s_tmem)),
                     "n"(kSelTmemCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    const uint32_t mbar = smem_addr(&s_mbar);
    if (tid == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(mbar));
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = s_tmem;

    const uint32_t sbase = smem_addr(smem);
    float* sAhi = reinterpret_cast<float*>(smem + LY::a_hi);
    float* sAlo = reinterpret_cast<float*>(smem + LY::a_lo);
    float* sBhi = reinterpret_cast<float*>(smem + LY::b_hi);
    float* sBlo = reinterpret_cast<float*>(smem + LY::b_lo);
    const T* ucol = static_cast<const T*>(p.u) + (size_t)bk * D * L + (lv ? l : 0);
    // this thread's row of A (its step): row group tid / 8, row tid % 8
    const int arow = (tid / 8) * 128 + (tid % 8) * 16;  // bytes within a channel quad's block
    constexpr int AG = kSelThreads / 8, BG = kSelCols / 8;
    bool ok = true;
    uint32_t phase = 0;
    // The tensor cores accumulate a run of kSelDrain chunks in TMEM; each run's
    // sums are then added to fp32 registers, which keeps the accumulation chain
    // inside the tensor cores short for wide maps (D up to 1536).
    float acc[kSelCols];
#pragma unroll
    for (int j = 0; j < kSelCols; ++j) acc[j] = 0.0f;
    auto drain = [&]() {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
        for (int c0 = 0; c0 < kSelCols; c0 += 16) {
            uint32_t r[16];
            const uint32_t taddr = tmem + ((uint32_t)(32 * warp) << 16) + (uint32_t)c0;
            asm volatile(
                "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, "
                "[%16];"
                : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
                  "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
                : "r"(taddr));
            asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
            for (int j = 0; j < 16; ++j) acc[c0 + j] += __uint_as_float(r[j]);
        }
        // the next run's first MMA overwrites the accumulator only after every warp has read it
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();
    };
    const int nchunks = (D + kSelKC - 1) / kSelKC;
    // u of this step over a chunk's channels (coalesced across the steps of a
    // warp) and this thread's share of the chunk's weights (B rows 0..15, C rows
    // 16..31, z rows 32..47, zero past N / R / D), all loads in flight
    // together; the next chunk's loads are issued while the tensor cores work
    // on the current one
    constexpr int kWPT = kSelCols * kSelKC / kSelThreads;  // weights per thread and chunk
    float v[kSelKC], wv[kWPT];
    auto load_chunk = [&](int c0) {
        const int cn = min(kSelKC, D - c0);
#pragma unroll
        for (int j = 0; j < kSelKC; ++j) v[j] = (lv && j < cn) ? io<T>::ld(ucol + (size_t)(c0 + j) * L) : 0.0f;
#pragma unroll
        for (int q = 0; q < kWPT; ++q) {
            const int i = tid + q * kSelThreads, m = i / kSelKC, j = i % kSelKC;
            const float* src = m < 16 ? p.WB + ((size_t)k * N + m) * D
                                      : m < 32 ? p.WC + ((size_t)k * N + (m - 16)) * D
                                               : p.Wz + ((size_t)k * R + (m - 32)) * D;
            const bool in = j < cn && (m < 16 ? m < N : m < 32 ? m - 16 < N : m - 32 < R);
            wv[q] = in ? __ldg(src + c0 + j) : 0.0f;
        }
    };
    load_chunk(0);
    for (int chunk = 0; chunk < nchunks; ++chunk) {
        const int d0 = chunk * kSelKC;
        const int dn = min(kSelKC, D - d0);
#pragma unroll
        for (int c = 0; c < kSelKC / 4; ++c) {
            float hi[4], lo[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                hi[e] = F32 ? to_tf32(v[4 * c + e]) : v[4 * c + e];  // bf16 values are exact in tf32
                lo[e] = to_tf32(v[4 * c + e] - hi[e]);
            }
            const int off = (c * AG * 128 + arow) / 4;
            *reinterpret_cast<float4*>(sAhi + off) = make_float4(hi[0], hi[1], hi[2], hi[3]);
            if constexpr (F32) *reinterpret_cast<float4*>(sAlo + off) = make_float4(lo[0], lo[1], lo[2], lo[3]);
        }
        // the chunk's weight rows in the same layout
#pragma unroll
        for (int q = 0; q < kWPT; ++q) {
            const int i = tid + q * kSelThreads, m = i / kSelKC, j = i % kSelKC;
            const float hi = to_tf32(wv[q]);
            const int off = ((j / 4) * BG * 128 + (m / 8) * 128 + (m % 8) * 16) / 4 + (j % 4);
            sBhi[off] = hi;
            sBlo[off] = to_tf32(wv[q] - hi);
        }
        // the generic-proxy stores become visible to the tensor cores' async proxy
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        if (tid == 0) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const int ksteps = (dn + 7) / 8;
            for (int ks = 0; ks < ksteps; ++ks) {
                // k-step ks covers channel quads 2 ks and 2 ks + 1
                const uint32_t ao = (uint32_t)(2 * ks * AG * 128), bo = (uint32_t)(2 * ks * BG * 128);
                const uint64_t ahi = mma_desc(sbase + (uint32_t)LY::a_hi + ao, AG * 128, 128);
                const uint64_t bhi = mma_desc(sbase + (uint32_t)LY::b_hi + bo, BG * 128, 128);
                const uint64_t blo = mma_desc(sbase + (uint32_t)LY::b_lo + bo, BG * 128, 128);
                mma_tf32(tmem, ahi, bhi, (chunk % kSelDrain != 0 || ks > 0) ? 1u : 0u);
                mma_tf32(tmem, ahi, blo, 1u);
                if constexpr (F32) {
                    const uint64_t alo = mma_desc(sbase + (uint32_t)LY::a_lo + ao, AG * 128, 128);
                    mma_tf32(tmem, alo, bhi, 1u);
                }
            }
            asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(mbar)
                         : "memory");
        }
        if (chunk + 1 < nchunks) load_chunk(d0 + kSelKC);
        // the chunk's MMAs have read the operands before they are overwritten
        // (after a wait that gave up, the rest of the tile is not waited for)
        if (ok) ok = mbar_wait(mbar, phase);
        phase ^= 1u;
        // this step's sums of the run: warp w reads TMEM lanes 32 w .. 32 w + 31
        if (chunk % kSelDrain == kSelDrain - 1 || chunk == nchunks - 1) drain();
    }
    if (!ok) {
#pragma unroll
        for (int j = 0; j < kSelCols; ++j) acc[j] = __int_as_float(0x7fffffff);  // a wait gave up: NaN outputs
    }
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(kSelTmemCols));

    if (lv) {
        T* ob = static_cast<T*>(p.Bs) + (size_t)bk * N * L + l;
        T* oc = static_cast<T*>(p.Cs) + (size_t)bk * N * L + l;
#pragma unroll
        for (int n = 0; n < 16; ++n) {
            if (n < N) {
                ob[(size_t)n * L] = io<T>::to(acc[n]);
                oc[(size_t)n * L] = io<T>::to(acc[16 + n]);
            }
        }
    }
    if (p.z) {
        // the low-rank form: z itself, for a scan that expands it through Wup
        if (lv) {
            float* oz = p.z + (size_t)bk * R * L + l;
#pragma unroll
            for (int r = 0; r < 16; ++r)
                if (r < R) oz[(size_t)r * L] = acc[32 + r];
        }
        return;
    }
    // the raw Deltas: z expanded through Wup, kSelDB channels' rows staged at a
    // time over the operand area (rows padded to kSelRP with zeros)
    float* sW = reinterpret_cast<float*>(smem);
    T* od = static_cast<T*>(p.dr) + (size_t)bk * D * L + (lv ? l : 0);
    for (int c0 = 0; c0 < D; c0 += kSelDB) {
        const int cn = min(kSelDB, D - c0);
        __syncthreads();  // the previous rows are no longer read
        for (int i = tid; i < kSelDB * kSelRP; i += kSelThreads) {
            const int j = i / kSelRP, r = i % kSelRP;
            sW[i] = (j < cn && r < R) ? __ldg(p.Wup + ((size_t)k * D + c0 + j) * R + r) : 0.0f;
        }
        __syncthreads();
        if (lv) {
#pragma unroll 4
            for (int j = 0; j < cn; ++j) {
                const float4* w4 = reinterpret_cast<const float4*>(sW + j * kSelRP);
                float s = 0.0f;
#pragma unroll
                for (int q = 0; q < kSelRP / 4; ++q) {
                    if (4 * q < R) {
                        const float4 w = w4[q];
                        s = fmaf(w.x, acc[32 + 4 * q], s);
                        s = fmaf(w.y, acc[33 + 4 * q], s);
                        s = fmaf(w.z, acc[34 + 4 * q], s);
                        s = fmaf(w.w, acc[35 + 4 * q], s);
                    }
                }
                od[(size_t)(c0 + j) * L] = io<T>::to(s);
            }
        }
    }
}

template <typename T>
const void* sel_fn() {
    const void* fn = reinterpret_cast<const void*>(&selection_kernel<T>);
    static std::once_flag once;
    static cudaError_t err = cudaSuccess;
    std::call_once(once, [&] {
        err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SelLayout::bytes);
    });
    return err == cudaSuccess ? fn : nullptr;
}

}  // namespace

vmb_status launch_selection(const SelArgs& a, cudaStream_t stream) {
    SelParams p{};
    p.u = a.u;
    p.WB = a.WB;
    p.WC = a.WC;
    p.Wz = a.Wz;
    p.Wup = a.Wup;
    p.Bs = a.Bs;
    p.Cs = a.Cs;
    p.dr = a.delta_raw;
    p.z = a.z;
    p.K = a.K;
    p.D = a.D;
    p.N = a.N;
    p.R = a.R;
    p.L = a.L;
    p.nlb = (a.L + kSelThreads - 1) / kSelThreads;
    const long long grid = (long long)a.B * a.K * p.nlb;
    if (grid > INT32_MAX) return VMB_ERR_UNSUPPORTED;
    const void* fn = a.dtype == VMB_BF16 ? sel_fn<__nv_bfloat16>() : sel_fn<float>();
    if (!fn) return VMB_ERR_CUDA;
    void* args[] = {&p};
    return launch_kernel(fn, dim3((unsigned)grid), dim3(kSelThreads), SelLayout::bytes, args, stream) == cudaSuccess
               ? VMB_OK
               : VMB_ERR_CUDA;
}

}  // namespace vmb
