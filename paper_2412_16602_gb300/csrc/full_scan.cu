// full_scan.cu - full-channel selective scan (App. A, Eqs. 3, 4, 6) for sm_103a.
//
// One CTA owns a tile of DT channels of one (batch, direction) and one chunk
// of the sequence.  G adjacent lanes share a channel, each owning NG = NP/G of
// its NP states (G = 1, 2 or 4, picked by the planner from the available row
// parallelism).  The chunk streams through shared memory in stages of TS
// steps (cp.async, double buffered, u and delta rows padded so that the
// per-channel 128-bit reads are free of bank conflicts).  In registers, per
// step: delta = softplus(raw + bias) (Eq. 6, computed once per element, the G
// lanes of a channel splitting the steps and sharing by shuffle), Abar =
// 2^(delta A log2 e) on the MUFU pipe, Bbar u = delta u B (Eq. 4), h = Abar h
// + Bbar u and y = C.h + D u (Eq. 3).  B and C are transposed to [t][n] per stage so a lane
// reads its states as 128-bit vectors.  y is reduced across the G lanes by a
// transposed butterfly, staged in shared memory and written with 16-byte
// stores.
//
// Long sequences with few channels are cut into L-chunks that run in
// parallel.  Chunks after the first run twice: a first pass computes the
// chunk's aggregate (S = sum of delta, so prod Abar_n = 2^(A_n log2 e S), and
// H = end state from h = 0) and publishes it; a decoupled look-back finds the
// carry-in state; the second pass recomputes the chunk from that state and
// writes y.  Chunk order follows a ticket counter, so a CTA only waits on
// CTAs that started before it; every wait is bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>
#include <type_traits>

#include "vmb_common.cuh"
#include "vmb_internal.h"

namespace vmb {
namespace {

struct FullParams {
    const void* u;
    const void* dl;
    const float* A;
    const void* Bs;
    const void* Cs;
    const float* Dskip;
    const float* bias;
    void* y;
    int K, D, N, L;
    int softplus_on;
    int tiles_per_bk, n_tiles, n_chunks, chunk_len;
    int vec;       // rows are 16-byte aligned: cp.async 16-byte path and vector stores
    int suppress;  // test hook: chunk 0 does not publish
    int gather_h;  // > 0: u is gathered from the map x and its transpose (warp-specialised variant only)
    const float* Wup;  // low-rank Delta (warp-specialised variant only): dl is z [B*K][R][L] fp32 and
    int R;             // delta_raw[b,k,d,l] = sum_r Wup[k,d,r] z[b,k,r,l]
    WsHeader* hdr;
    unsigned* flags;
    float* aggP;   // per chunk: sum of delta per channel (DT floats, rest unused)
    float* aggH;
    float* incH;
};

__host__ __device__ constexpr size_t a16(size_t v) { return (v + 15) / 16 * 16; }

// Tile shape: G lanes per channel, DT channels per CTA, TS steps per stage
// (0: one 16-byte chunk per row), NSTG stages in the cp.async ring, and the
// CTAs per SM the register budget is sized for.
template <int G_, int DT_, int TS_, int NSTG_, int MINB_ = 1>
struct Shape {
    static constexpr int G = G_, DT = DT_, TS = TS_, NSTG = NSTG_, MINB = MINB_;
};

template <typename T, int NP, class SH>
struct Layout {
    static constexpr int G = SH::G, DT = SH::DT, NSTG = SH::NSTG, MINB = SH::MINB;
    static constexpr int TS = SH::TS ? SH::TS : 16 / (int)sizeof(T);
    static constexpr int THREADS = DT * G;
    static constexpr int PAD = 16 / (int)sizeof(T);  // one 16-byte chunk of row padding
    static constexpr int RS = TS + PAD;               // raw row stride (elements)
    static constexpr int SLOT = (2 * DT + 2 * NP) * RS;
    static constexpr size_t raw_bytes = a16((size_t)NSTG * SLOT * sizeof(T));
    static constexpr size_t bf_off = raw_bytes;                      // 2 slots of [TS][NP] fp32
    static constexpr size_t cf_off = bf_off + (size_t)2 * TS * NP * 4;
    static constexpr size_t bytes = cf_off + (size_t)2 * TS * NP * 4;
    static_assert(TS % 4 == 0 && NP % G == 0 && THREADS % 32 == 0 && NSTG >= 3, "tile shape");
    static_assert(bytes <= 100 * 1024, "full-scan tile must leave room for two CTAs per SM");
};

// Four consecutive elements of one row as fp32 (16-byte / 8-byte aligned reads).
__device__ __forceinline__ void load4(const float* p, float (&v)[4]) {
    const float4 q = *reinterpret_cast<const float4*>(p);
    v[0] = q.x;
    v[1] = q.y;
    v[2] = q.z;
    v[3] = q.w;
}
__device__ __forceinline__ void load4(const __nv_bfloat16* p, float (&v)[4]) {
    const uint2 q = *reinterpret_cast<const uint2*>(p);
    v[0] = __uint_as_float(q.x << 16);
    v[1] = __uint_as_float(q.x & 0xffff0000u);
    v[2] = __uint_as_float(q.y << 16);
    v[3] = __uint_as_float(q.y & 0xffff0000u);
}

// NG consecutive fp32 values from shared memory (16-byte aligned when NG >= 4).
template <int NG>
__device__ __forceinline__ void load_states(const float* p, float (&v)[NG]) {
    if constexpr (NG % 4 == 0) {
#pragma unroll
        for (int i = 0; i < NG; i += 4) {
            const float4 q = *reinterpret_cast<const float4*>(p + i);
            v[i] = q.x;
            v[i + 1] = q.y;
            v[i + 2] = q.z;
            v[i + 3] = q.w;
        }
    } else {
#pragma unroll
        for (int i = 0; i < NG; ++i) v[i] = p[i];
    }
}

__device__ __forceinline__ float sel4(const float (&v)[4], int j) {
    return j == 0 ? v[0] : j == 1 ? v[1] : j == 2 ? v[2] : v[3];
}

// Store n consecutive outputs of one row (n = 4, 2 or 1), vectorised when aligned.
template <typename T, int NV>
__device__ __forceinline__ void store_row(T* dst, const float (&v)[NV], int nvalid_here, bool vec) {
    if (vec && nvalid_here >= NV) {
        if constexpr (sizeof(T) == 4 && NV == 4) {
            *reinterpret_cast<float4*>(dst) = make_float4(v[0], v[1], v[2], v[3]);
            return;
        } else if constexpr (sizeof(T) == 4 && NV == 2) {
            *reinterpret_cast<float2*>(dst) = make_float2(v[0], v[1]);
            return;
        } else if constexpr (sizeof(T) == 2 && NV == 4) {
            const unsigned lo = __bfloat16_as_ushort(io<T>::to(v[0])) | ((unsigned)__bfloat16_as_ushort(io<T>::to(v[1])) << 16);
            const unsigned hi = __bfloat16_as_ushort(io<T>::to(v[2])) | ((unsigned)__bfloat16_as_ushort(io<T>::to(v[3])) << 16);
            *reinterpret_cast<uint2*>(dst) = make_uint2(lo, hi);
            return;
        } else if constexpr (sizeof(T) == 2 && NV == 2) {
            *reinterpret_cast<unsigned*>(dst) =
                __bfloat16_as_ushort(io<T>::to(v[0])) | ((unsigned)__bfloat16_as_ushort(io<T>::to(v[1])) << 16);
            return;
        }
    }
#pragma unroll
    for (int j = 0; j < NV; ++j)
        if (j < nvalid_here) dst[j] = io<T>::to(v[j]);
}

// Copy kTS steps (from l0) of DT u and delta rows and of the NP B (and C) rows
// into shared memory rows of stride RS: u at row 0, delta at row DT, B at 2 DT,
// C at 2 DT + NP.  Rows and steps past the problem are zero-filled.
template <typename T, int NP, int DT, int kTS, int RS, int kThreads, bool WITH_C, bool WITH_B = true>
__device__ __forceinline__ void load_tile(const FullParams& p, T* dst, size_t row0, size_t bcrow0, int nrows,
                                          int l0) {
    constexpr int VE = 16 / sizeof(T);  // elements per 16-byte chunk
    constexpr int CPR = kTS / VE;       // chunks per stage row
    static_assert(kTS % VE == 0, "a stage row is a whole number of 16-byte chunks");
    const T* u = static_cast<const T*>(p.u);
    const T* dl = static_cast<const T*>(p.dl);
    const T* Bs = static_cast<const T*>(p.Bs);
    const T* Cs = static_cast<const T*>(p.Cs);
    const int L = p.L;
    T* dB = dst + 2 * DT * RS;
    if (p.vec) {
        // thread i copies 16-byte column i % CPR of rows i / CPR + k * RPP
        constexpr int RPP = kThreads / CPR;  // rows covered per pass of the CTA
        static_assert(kThreads % CPR == 0, "tile loader mapping");
        const int ch = threadIdx.x % CPR, r0 = threadIdx.x / CPR;
        const int col = l0 + ch * VE;
        const bool colok = col < L;
#pragma unroll
        for (int it = 0; it < (DT + RPP - 1) / RPP; ++it) {
            const int r = r0 + it * RPP;
            if (DT % RPP == 0 || r < DT) {
                const bool ok = colok && r < nrows;
                const size_t off = (row0 + r) * (size_t)L + col;
                cp_async16(dst + r * RS + ch * VE, ok ? u + off : u, ok ? 16 : 0);
                cp_async16(dst + (DT + r) * RS + ch * VE, ok ? dl + off : dl, ok ? 16 : 0);
            }
        }
        if constexpr (WITH_B) {
#pragma unroll
            for (int it = 0; it < (NP + RPP - 1) / RPP; ++it) {
                const int r = r0 + it * RPP;
                if (r < NP) {
                    const bool ok = colok && r < p.N;
                    const size_t off = (bcrow0 + r) * (size_t)L + col;
                    cp_async16(dB + r * RS + ch * VE, ok ? Bs + off : Bs, ok ? 16 : 0);
                    if constexpr (WITH_C) cp_async16(dB + (NP + r) * RS + ch * VE, ok ? Cs + off : Cs, ok ? 16 : 0);
                }
            }
        }
    } else {
        constexpr int nU = DT * kTS, nB = NP * kTS;
        constexpr int total = 2 * nU + (WITH_B ? (WITH_C ? 2 : 1) * nB : 0);
        for (int i = threadIdx.x; i < total; i += kThreads) {
            T v = T(0.0f);
            if (i < 2 * nU) {
                const int j = i < nU ? i : i - nU;
                const int r = j / kTS, t = j % kTS;
                const T* base = i < nU ? u : dl;
                if (r < nrows && l0 + t < L) v = base[(row0 + r) * (size_t)L + l0 + t];
                dst[(i < nU ? 0 : DT * RS) + r * RS + t] = v;
            } else {
                const int i2 = i - 2 * nU;
                const int j = i2 < nB ? i2 : i2 - nB;
                const int r = j / kTS, t = j % kTS;
                const T* base = i2 < nB ? Bs : Cs;
                if (r < p.N && l0 + t < L) v = base[(bcrow0 + r) * (size_t)L + l0 + t];
                dB[(i2 < nB ? 0 : NP * RS) + r * RS + t] = v;
            }
        }
    }
}

template <typename T, int NP, class SH, bool WITH_C>
__device__ __forceinline__ void load_stage(const FullParams& p, T* dst, size_t row0, size_t bcrow0, int nrows,
                                           int l0) {
    using LY = Layout<T, NP, SH>;
    load_tile<T, NP, LY::DT, LY::TS, LY::RS, LY::THREADS, WITH_C>(p, dst, row0, bcrow0, nrows, l0);
}

template <typename T, int NP, class SH, bool ZOH>
__global__ void __launch_bounds__(Layout<T, NP, SH>::THREADS, Layout<T, NP, SH>::MINB)
    full_scan_kernel(const FullParams p) {
    pdl_wait();
    pdl_launch_dependents();
    using LY = Layout<T, NP, SH>;
    constexpr int kThreads = LY::THREADS, kTS = LY::TS, RS = LY::RS, SLOT = LY::SLOT, DT = LY::DT;
    constexpr int G = LY::G, NSTG = LY::NSTG;
    constexpr int NG = NP / G;
    extern __shared__ __align__(16) unsigned char smem[];
    T* raw = reinterpret_cast<T*>(smem);
    float* bfm = reinterpret_cast<float*>(smem + LY::bf_off);
    float* cfm = reinterpret_cast<float*>(smem + LY::cf_off);
    __shared__ unsigned s_misc[2];

    const int tid = threadIdx.x;
    int tile, chunk;
    unsigned gen = 0;
    const bool chunked = p.n_chunks > 1;
    if (chunked) {
        if (tid == 0) {
            s_misc[0] = atomicAdd(&p.hdr->ticket, 1u);
            s_misc[1] = ld_relaxed(&p.hdr->gen);
        }
        __syncthreads();
        const unsigned t = s_misc[0];
        gen = s_misc[1];
        if (t >= (unsigned)(p.n_tiles * p.n_chunks)) {  // workspace was not zero-filled
            if (tid == 0) {
                atomicOr(&p.hdr->err, kErrBounds);
                finish_launch(p.hdr, (unsigned)(p.n_tiles * p.n_chunks));
            }
            return;
        }
        chunk = (int)(t / (unsigned)p.n_tiles);
        tile = (int)(t % (unsigned)p.n_tiles);
    } else {
        tile = blockIdx.x;
        chunk = 0;
    }
    const int bk = tile / p.tiles_per_bk;
    const int d0 = (tile % p.tiles_per_bk) * DT;
    const int k = bk % p.K;
    const int c = tid / G, g = tid % G;
    const int d = d0 + c;
    const bool cval = d < p.D;
    const int nrows = min(DT, p.D - d0);
    const size_t row0 = (size_t)bk * p.D + d0;
    const size_t bcrow0 = (size_t)bk * p.N;

    float A2[NG], Ar[NG], h[NG];
#pragma unroll
    for (int i = 0; i < NG; ++i) {
        const int n = g * NG + i;
        const float a = (cval && n < p.N) ? p.A[((size_t)k * p.D + d) * p.N + n] : 0.0f;
        A2[i] = a * kLog2e;
        Ar[i] = a;
        h[i] = 0.0f;
    }
    const float dsk = cval ? p.Dskip[(size_t)k * p.D + d] : 0.0f;
    const float bias = cval ? p.bias[(size_t)k * p.D + d] : 0.0f;
    const int l_begin = chunk * p.chunk_len;
    const int l_end = min(p.L, l_begin + p.chunk_len);
    const int nst = (l_end - l_begin + kTS - 1) / kTS;
    T* yrow = static_cast<T*>(p.y) + (row0 + c) * (size_t)p.L;
    float ssum = 0.0f;  // sum of delta over the chunk (first pass)

    // One pass over the chunk.  PH2 = false: aggregate only (h from 0, S).
    // PH2 = true: recurrence from the carried-in h, output y.
    // Ring of NSTG raw stages, prefetch distance NSTG - 1; B and C of stage s+1
    // are transposed to [t][n] while stage s is computed; one barrier per stage.
    // Steps past the end of the sequence (last stage only) run on zero-filled
    // inputs; their outputs are not stored and the final state is not used.
    auto pass = [&](auto ph2_tag) {
        constexpr bool PH2 = decltype(ph2_tag)::value;
        auto transpose = [&](int st) {
            const T* rb = raw + (st % NSTG) * SLOT + 2 * DT * RS;
            const T* rc = rb + NP * RS;
            float* bo = bfm + (st & 1) * kTS * NP;
            float* co = cfm + (st & 1) * kTS * NP;
            for (int i = tid; i < NP * kTS; i += kThreads) {
                const int n = i % NP, t = i / NP;
                bo[t * NP + n] = io<T>::cvt(rb[n * RS + t]);
                if constexpr (PH2) co[t * NP + n] = io<T>::cvt(rc[n * RS + t]);
            }
        };
#pragma unroll
        for (int q = 0; q < NSTG - 1; ++q) {
            if (q < nst) load_stage<T, NP, SH, PH2>(p, raw + q * SLOT, row0, bcrow0, nrows, l_begin + q * kTS);
            cp_async_commit();
        }
        cp_async_wait<NSTG - 2>();
        __syncthreads();
        transpose(0);
        for (int s = 0; s < nst; ++s) {
            const int l0 = l_begin + s * kTS;
            const int nvalid = min(kTS, l_end - l0);
            cp_async_wait<NSTG - 3>();  // stages <= s+1 have landed
            __syncthreads();
            if (s + NSTG - 1 < nst)
                load_stage<T, NP, SH, PH2>(p, raw + ((s + NSTG - 1) % NSTG) * SLOT, row0, bcrow0, nrows,
                                           l0 + (NSTG - 1) * kTS);
            cp_async_commit();
            if (s + 1 < nst) transpose(s + 1);
            const T* ru = raw + (s % NSTG) * SLOT;
            const T* rd = ru + DT * RS;
            const float* bst = bfm + (s & 1) * kTS * NP;
            const float* cst = cfm + (s & 1) * kTS * NP;
#pragma unroll 1
            for (int t0 = 0; t0 < kTS; t0 += 4) {
                float u4[4], r4[4], dl4[4];
                load4(ru + c * RS + t0, u4);
                load4(rd + c * RS + t0, r4);
                // softplus once per element; the G lanes of a channel split the steps
                if constexpr (G == 1) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float v = r4[j] + bias;
                        dl4[j] = p.softplus_on ? softplus(v) : v;
                    }
                } else if constexpr (G == 2) {
                    const float va = (g ? r4[1] : r4[0]) + bias, vb = (g ? r4[3] : r4[2]) + bias;
                    const float a = p.softplus_on ? softplus(va) : va;
                    const float b = p.softplus_on ? softplus(vb) : vb;
                    const float oa = __shfl_xor_sync(0xffffffffu, a, 1);
                    const float ob = __shfl_xor_sync(0xffffffffu, b, 1);
                    dl4[0] = g ? oa : a;
                    dl4[1] = g ? a : oa;
                    dl4[2] = g ? ob : b;
                    dl4[3] = g ? b : ob;
                } else {
                    const float v = sel4(r4, g) + bias;
                    const float a = p.softplus_on ? softplus(v) : v;
                    const int base = (threadIdx.x & 31) & ~3;
#pragma unroll
                    for (int j = 0; j < 4; ++j) dl4[j] = __shfl_sync(0xffffffffu, a, base + j);
                }
                float yp[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int t = t0 + j;
                    const float dlt = dl4[j];
                    const float uu = u4[j];
                    if constexpr (!PH2) ssum += (t < nvalid) ? dlt : 0.0f;
                    const float du = dlt * uu;
                    float Bv[NG], Cv[NG];
                    load_states<NG>(bst + t * NP + g * NG, Bv);
                    if constexpr (PH2) load_states<NG>(cst + t * NP + g * NG, Cv);
                    // scalar FP32 (on GB300 the packed f32x2 forms issue slower in this
                    // MUFU-heavy mix); four accumulators keep the y chain short
                    float ya[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
                    for (int i = 0; i < NG; ++i) {
                        float a, bb;
                        if constexpr (ZOH) {
                            const float em1 = expm1f(dlt * Ar[i]);
                            a = 1.0f + em1;
                            bb = (Ar[i] != 0.0f ? em1 / Ar[i] : dlt) * Bv[i] * uu;
                        } else {
                            a = ex2(dlt * A2[i]);
                            bb = du * Bv[i];
                        }
                        h[i] = fmaf(a, h[i], bb);
                        if constexpr (PH2) ya[i & 3] = fmaf(Cv[i], h[i], ya[i & 3]);
                    }
                    yp[j] = (ya[0] + ya[1]) + (ya[2] + ya[3]);
                }
                if constexpr (PH2) {
                    // y = sum over the channel's lanes + D u, stored straight from registers
                    if constexpr (G == 1) {
                        float o[4];
#pragma unroll
                        for (int j = 0; j < 4; ++j) o[j] = fmaf(dsk, u4[j], yp[j]);
                        if (cval) store_row<T, 4>(yrow + l0 + t0, o, nvalid - t0, p.vec);
                    } else if constexpr (G == 2) {
                        // lane g keeps steps 2g and 2g+1
                        const float k0 = g ? yp[2] : yp[0], k1 = g ? yp[3] : yp[1];
                        const float s0 = g ? yp[0] : yp[2], s1 = g ? yp[1] : yp[3];
                        float o[2];
                        o[0] = fmaf(dsk, g ? u4[2] : u4[0], k0 + __shfl_xor_sync(0xffffffffu, s0, 1));
                        o[1] = fmaf(dsk, g ? u4[3] : u4[1], k1 + __shfl_xor_sync(0xffffffffu, s1, 1));
                        if (cval) store_row<T, 2>(yrow + l0 + t0 + 2 * g, o, nvalid - t0 - 2 * g, p.vec);
                    } else {
                        const bool hi = g & 2;
                        float k0 = hi ? yp[2] : yp[0], k1 = hi ? yp[3] : yp[1];
                        const float s0 = hi ? yp[0] : yp[2], s1 = hi ? yp[1] : yp[3];
                        k0 += __shfl_xor_sync(0xffffffffu, s0, 2);
                        k1 += __shfl_xor_sync(0xffffffffu, s1, 2);
                        const bool odd = g & 1;
                        const float kk = odd ? k1 : k0, ss = odd ? k0 : k1;
                        float o[1];
                        o[0] = fmaf(dsk, sel4(u4, g), kk + __shfl_xor_sync(0xffffffffu, ss, 1));
                        if (cval) store_row<T, 1>(yrow + l0 + t0 + g, o, nvalid - t0 - g, false);
                    }
                }
            }
        }
        cp_async_wait<0>();
        __syncthreads();
    };

    const size_t sfl = (size_t)DT * NP;  // floats of one published state
    const size_t my_off = (size_t)c * NP + (size_t)g * NG;
    if (chunked && chunk > 0) {
        pass(std::false_type{});
        const size_t slot = (size_t)tile * p.n_chunks + chunk;
        if (g == 0) p.aggP[slot * sfl + c] = ssum;
#pragma unroll
        for (int i = 0; i < NG; ++i) p.aggH[slot * sfl + my_off + i] = h[i];
        __threadfence();
        __syncthreads();
        if (tid == 0) st_release(&p.flags[slot], flag_word(gen, kFlagAggregate));
        // Decoupled look-back: walk back until a predecessor's inclusive state is
        // published, then fold the aggregates after it left to right,
        // h <- 2^(A_n log2 e S_m) h + H_m.  Every inclusive state is defined by
        // this same left fold from chunk 0, so the carry is bit-identical
        // whichever predecessor the walk stops at (results do not depend on
        // scheduling).
        if (tid < 32) {
            const int f = lookback_find(p.flags + (size_t)tile * p.n_chunks, chunk, gen, p.hdr, (unsigned)tile);
            if (tid == 0) s_misc[0] = (unsigned)f;
        }
        __syncthreads();
        const int found = (int)s_misc[0];
        float RH[NG];
#pragma unroll
        for (int i = 0; i < NG; ++i) RH[i] = 0.0f;
        if (found >= 0) {
            const size_t sf = (size_t)tile * p.n_chunks + found;
#pragma unroll
            for (int i = 0; i < NG; ++i) RH[i] = ld_cg(&p.incH[sf * sfl + my_off + i]);
            for (int m = found + 1; m < chunk; ++m) {
                const size_t sm = (size_t)tile * p.n_chunks + m;
                const float sm_s = ld_cg(&p.aggP[sm * sfl + c]);
#pragma unroll
                for (int i = 0; i < NG; ++i)
                    RH[i] = fmaf(ex2(A2[i] * sm_s), RH[i], ld_cg(&p.aggH[sm * sfl + my_off + i]));
            }
        }
        // inclusive end state of this chunk
#pragma unroll
        for (int i = 0; i < NG; ++i) {
            p.incH[slot * sfl + my_off + i] = fmaf(ex2(A2[i] * ssum), RH[i], h[i]);
            h[i] = RH[i];
        }
        __threadfence();
        __syncthreads();
        if (tid == 0) st_release(&p.flags[slot], flag_word(gen, kFlagInclusive));
    }

    pass(std::true_type{});

    if (chunked) {
        if (chunk == 0) {
            const size_t slot = (size_t)tile * p.n_chunks;
#pragma unroll
            for (int i = 0; i < NG; ++i) p.incH[slot * sfl + my_off + i] = h[i];
            __threadfence();
            __syncthreads();
            if (tid == 0 && !p.suppress) st_release(&p.flags[slot], flag_word(gen, kFlagInclusive));
        }
        __syncthreads();
        if (tid == 0) finish_launch(p.hdr, (unsigned)(p.n_tiles * p.n_chunks));
    }
}

// ----------------------------------------------------------- lane-per-state variant
// For problems with few channel rows (a batch-1 map): the 16 lanes of a
// half-warp share one channel and each owns one of its 16 states, so a channel
// row gets 16x the threads of the one-lane-per-channel tiles and a long
// sequence needs few or no L-chunks.  Per step a lane does one state update;
// delta and delta*u are computed once per step by one lane of the channel and
// broadcast by shuffle; B and C are read from the stage rows as they landed
// ([n][t], four steps per 128-bit read, no transpose); y is reduced over the 16
// lanes by a transposed butterfly every 16 steps (lane n ends with step t0+n).
using LanesShape = Shape<16, 16, 32, 3>;  // 16 lanes per channel, 16 channels, 32-step stages

// Sum of v[0..CNT) over the lanes of a half-warp, transposed: after the four
// levels lane n holds the sum for index n.
template <int CNT, int M>
__device__ __forceinline__ void reduce_level(float (&v)[16], bool up) {
#pragma unroll
    for (int i = 0; i < CNT / 2; ++i) {
        const float keep = up ? v[i + CNT / 2] : v[i];
        const float send = up ? v[i] : v[i + CNT / 2];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, M);
    }
}

template <typename T, bool ZOH>
__global__ void __launch_bounds__(256) full_scan_lanes_kernel(const FullParams p) {
    pdl_wait();
    pdl_launch_dependents();
    using LY = Layout<T, 16, LanesShape>;
    constexpr int kTS = LY::TS, RS = LY::RS, SLOT = LY::SLOT, DT = LY::DT, NSTG = LY::NSTG;
    extern __shared__ __align__(16) unsigned char smem[];
    T* raw = reinterpret_cast<T*>(smem);
    __shared__ unsigned s_misc[2];

    const int tid = threadIdx.x;
    int tile, chunk;
    unsigned gen = 0;
    const bool chunked = p.n_chunks > 1;
    if (chunked) {
        if (tid == 0) {
            s_misc[0] = atomicAdd(&p.hdr->ticket, 1u);
            s_misc[1] = ld_relaxed(&p.hdr->gen);
        }
        __syncthreads();
        const unsigned t = s_misc[0];
        gen = s_misc[1];
        if (t >= (unsigned)(p.n_tiles * p.n_chunks)) {  // workspace was not zero-filled
            if (tid == 0) {
                atomicOr(&p.hdr->err, kErrBounds);
                finish_launch(p.hdr, (unsigned)(p.n_tiles * p.n_chunks));
            }
            return;
        }
        chunk = (int)(t / (unsigned)p.n_tiles);
        tile = (int)(t % (unsigned)p.n_tiles);
    } else {
        tile = blockIdx.x;
        chunk = 0;
    }
    const int bk = tile / p.tiles_per_bk;
    const int d0 = (tile % p.tiles_per_bk) * DT;
    const int k = bk % p.K;
    const int lane = tid & 31;
    const int c = (tid >> 5) * 2 + (lane >> 4);  // channel within the tile
    const int n = lane & 15;                     // state owned by this lane
    const int hb = lane & 16;                    // first lane of the channel's half-warp
    const int d = d0 + c;
    const bool cval = d < p.D;
    const int nrows = min(DT, p.D - d0);
    const size_t row0 = (size_t)bk * p.D + d0;
    const size_t bcrow0 = (size_t)bk * p.N;
    const float Ar = (cval && n < p.N) ? p.A[((size_t)k * p.D + d) * p.N + n] : 0.0f;
    const float A2 = Ar * kLog2e;
    const float dsk = cval ? p.Dskip[(size_t)k * p.D + d] : 0.0f;
    const float bias = cval ? p.bias[(size_t)k * p.D + d] : 0.0f;
    const int l_begin = chunk * p.chunk_len;
    const int l_end = min(p.L, l_begin + p.chunk_len);
    const int nst = (l_end - l_begin + kTS - 1) / kTS;
    T* yrow = static_cast<T*>(p.y) + (row0 + c) * (size_t)p.L;
    float h = 0.0f;
    float ssum = 0.0f;  // this lane's share of the chunk's sum of delta (first pass)

    auto pass = [&](auto ph2_tag) {
        constexpr bool PH2 = decltype(ph2_tag)::value;
#pragma unroll
        for (int q = 0; q < NSTG - 1; ++q) {
            if (q < nst) load_stage<T, 16, LanesShape, PH2>(p, raw + q * SLOT, row0, bcrow0, nrows, l_begin + q * kTS);
            cp_async_commit();
        }
        for (int s = 0; s < nst; ++s) {
            const int l0 = l_begin + s * kTS;
            const int nvalid = min(kTS, l_end - l0);
            cp_async_wait<NSTG - 2>();  // stage s has landed
            __syncthreads();
            if (s + NSTG - 1 < nst)
                load_stage<T, 16, LanesShape, PH2>(p, raw + ((s + NSTG - 1) % NSTG) * SLOT, row0, bcrow0, nrows,
                                                   l0 + (NSTG - 1) * kTS);
            cp_async_commit();
            const T* ru = raw + (s % NSTG) * SLOT + c * RS;
            const T* rd = ru + DT * RS;
            const T* rb = raw + (s % NSTG) * SLOT + 2 * DT * RS + n * RS;
            const T* rc = rb + 16 * RS;
#pragma unroll 1
            for (int g0 = 0; g0 < kTS; g0 += 16) {
                // this lane's own step g0 + n: delta and delta * u, once per element
                const bool tv = g0 + n < nvalid;  // ragged tail: identity step (a = 1, b = 0)
                const float uo = tv ? io<T>::cvt(ru[g0 + n]) : 0.0f;
                const float vo = io<T>::cvt(rd[g0 + n]) + bias;
                const float dlo = tv ? (p.softplus_on ? softplus(vo) : vo) : 0.0f;
                const float duo = dlo * uo;
                if constexpr (!PH2) ssum += dlo;
                float Bv[16], Cv[16], yp[16];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    float t4[4];
                    load4(rb + g0 + 4 * q, t4);
                    Bv[4 * q] = t4[0];
                    Bv[4 * q + 1] = t4[1];
                    Bv[4 * q + 2] = t4[2];
                    Bv[4 * q + 3] = t4[3];
                    if constexpr (PH2) {
                        load4(rc + g0 + 4 * q, t4);
                        Cv[4 * q] = t4[0];
                        Cv[4 * q + 1] = t4[1];
                        Cv[4 * q + 2] = t4[2];
                        Cv[4 * q + 3] = t4[3];
                    }
                }
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const float dl = __shfl_sync(0xffffffffu, dlo, hb + j);
                    float a, bb;
                    if constexpr (ZOH) {
                        const float uu = __shfl_sync(0xffffffffu, uo, hb + j);
                        const float em1 = expm1f(dl * Ar);
                        a = 1.0f + em1;
                        bb = (Ar != 0.0f ? em1 / Ar : dl) * Bv[j] * uu;
                    } else {
                        const float du = __shfl_sync(0xffffffffu, duo, hb + j);
                        a = ex2(dl * A2);
                        bb = du * Bv[j];
                    }
                    h = fmaf(a, h, bb);
                    if constexpr (PH2) yp[j] = Cv[j] * h;
                }
                if constexpr (PH2) {
                    const bool u8 = n & 8, u4 = n & 4, u2 = n & 2, u1 = n & 1;
                    reduce_level<16, 8>(yp, u8);
                    reduce_level<8, 4>(yp, u4);
                    reduce_level<4, 2>(yp, u2);
                    reduce_level<2, 1>(yp, u1);
                    if (cval && tv) yrow[l0 + g0 + n] = io<T>::to(fmaf(dsk, uo, yp[0]));
                }
            }
        }
        cp_async_wait<0>();
        __syncthreads();
    };

    constexpr size_t sfl = (size_t)DT * 16;  // floats of one published state
    const size_t my_off = (size_t)c * 16 + n;
    if (chunked && chunk > 0) {
        pass(std::false_type{});
        // the channel's sum of delta over the chunk: add the 16 lanes' shares
        float cs = ssum;
#pragma unroll
        for (int m = 8; m >= 1; m >>= 1) cs += __shfl_xor_sync(0xffffffffu, cs, m);
        const size_t slot = (size_t)tile * p.n_chunks + chunk;
        if (n == 0) p.aggP[slot * sfl + c] = cs;
        p.aggH[slot * sfl + my_off] = h;
        __threadfence();
        __syncthreads();
        if (tid == 0) st_release(&p.flags[slot], flag_word(gen, kFlagAggregate));
        // decoupled look-back and left fold, as in full_scan_kernel
        if (tid < 32) {
            const int f = lookback_find(p.flags + (size_t)tile * p.n_chunks, chunk, gen, p.hdr, (unsigned)tile);
            if (tid == 0) s_misc[0] = (unsigned)f;
        }
        __syncthreads();
        const int found = (int)s_misc[0];
        float RH = 0.0f;
        if (found >= 0) {
            // staged fold, as in full_scan_kernel
            constexpr int kAgg = DT * 16 + DT;
            constexpr int kFB = (int)((size_t)NSTG * SLOT * sizeof(T) / (kAgg * 4));
            float* sa = reinterpret_cast<float*>(raw);
            RH = ld_cg(&p.incH[((size_t)tile * p.n_chunks + found) * sfl + my_off]);
            for (int m0 = found + 1; m0 < chunk; m0 += kFB) {
                const int nb = min(kFB, chunk - m0);
                for (int i = tid; i < nb * kAgg; i += 256) {
                    const int q = i / kAgg, r = i % kAgg;
                    const size_t sm = (size_t)tile * p.n_chunks + m0 + q;
                    sa[i] = r < DT * 16 ? ld_cg(&p.aggH[sm * sfl + r]) : ld_cg(&p.aggP[sm * sfl + (r - DT * 16)]);
                }
                __syncthreads();
                for (int q = 0; q < nb; ++q)
                    RH = fmaf(ex2(A2 * sa[q * kAgg + DT * 16 + c]), RH, sa[q * kAgg + my_off]);
                __syncthreads();
            }
        }
        p.incH[slot * sfl + my_off] = fmaf(ex2(A2 * cs), RH, h);
        h = RH;
        __threadfence();
        __syncthreads();
        if (tid == 0) st_release(&p.flags[slot], flag_word(gen, kFlagInclusive));
    }

    pass(std::true_type{});

    if (chunked) {
        if (chunk == 0) {
            const size_t slot = (size_t)tile * p.n_chunks;
            p.incH[slot * sfl + my_off] = h;
            __threadfence();
            __syncthreads();
            if (tid == 0 && !p.suppress) st_release(&p.flags[slot], flag_word(gen, kFlagInclusive));
        }
        __syncthreads();
        if (tid == 0) finish_launch(p.hdr, (unsigned)(p.n_tiles * p.n_chunks));
    }
}

// ------------------------------------------------------ three-launch chunked variant
// For long sequences with few channel rows (a batch-1 map) the sequence is cut
// into many short chunks of CL steps and the carry between chunks is resolved
// by three launches instead of a look-back, so that no CTA waits on another:
//   1. every chunk but the last computes its aggregate (S = sum of delta and
//      H = end state from h = 0) from a tile holding the whole chunk in shared
//      memory;
//   2. one thread per (channel, state) folds the aggregates left to right,
//      inc_m = 2^(A_n log2 e S_m) inc_{m-1} + H_m (the fold that defines the
//      inclusive states of the look-back path, so both give the same bits);
//   3. every chunk reruns its steps from the carried-in state inc_{m-1}, Eq. 3,
//      and writes y.
// G lanes per channel (1 or 2) own 16 / G of its states each; B and C are read
// from fp32 [n][t] rows four steps at a time (broadcast reads, no transpose),
// so a step costs one 128-bit read per state and operand.
template <int G_, int DT_, int CL_, int NS_, int MINB_>
struct ChunkShape {
    static constexpr int G = G_, DT = DT_, CL = CL_, NS = NS_, MINB = MINB_;  // NS: load sub-stages per chunk
};

template <typename T, class CS>
struct ChunkLayout {
    static constexpr int G = CS::G, DT = CS::DT, CL = CS::CL, NS = CS::NS, SUB = CL / NS, MINB = CS::MINB, NP = 16;
    static constexpr int THREADS = G * DT, NG = NP / G;
    static constexpr int PAD = 16 / (int)sizeof(T);
    static constexpr int RS = CL + PAD;  // row stride (elements); rows start 16-byte aligned
    static constexpr int ROWS = 2 * DT;  // u, delta (B and C go to the fp32 area)
    static constexpr size_t raw_bytes = a16((size_t)ROWS * RS * sizeof(T));
    // fp32 delta after the softplus: in place of the raw delta rows for fp32
    // storage, a separate [DT][CL + 4] area for bf16
    static constexpr int FS = CL + 4;
    static constexpr bool F32 = sizeof(T) == 4;
    static constexpr size_t dl_off = F32 ? (size_t)DT * RS * 4 : raw_bytes;
    // B and C as fp32 rows [2 NP][FS], converted once at load time (for bf16
    // storage one conversion per element instead of one per element and channel)
    static constexpr size_t bc_off = F32 ? raw_bytes : raw_bytes + (size_t)DT * FS * 4;
    static constexpr size_t a2_off = bc_off + (size_t)2 * NP * FS * 4;
    // G = 1: A * log2 e per channel in shared memory, [DT][16] with the four
    // 16-byte quads of a row swizzled by (c >> 1) & 3 so that eight consecutive
    // channels read their quad q from distinct banks (in registers it would
    // not leave room for the 16 states); G = 2 keeps its 8 values in registers
    static constexpr size_t bytes = a2_off + (G == 1 ? (size_t)DT * NP * 4 : 0);
    static_assert(CL % NS == 0 && SUB % (4 * G) == 0 && DT % 32 == 0 && NS <= 4 && (G == 1 || G == 2),
                  "chunk tile shape");
    static_assert(sizeof(T) == 2 || RS == FS, "fp32 delta rows are rewritten in place");
};


// Load of sub-stage `part` (steps part*SUB .. part*SUB+SUB-1) of the u and
// delta rows of the chunk tile: thread i always copies 16-byte column i % CPR
// of rows i / CPR + k * (THREADS / CPR), so the addresses advance by a fixed
// row stride.  Rows that are not 16-byte aligned take the element-wise loader,
// all of it with part 0.
template <typename T, class CS>
__device__ __forceinline__ void load_chunk_part(const FullParams& p, T* dst, size_t row0, int nrows, int l0,
                                                int part) {
    using LY = ChunkLayout<T, CS>;
    constexpr int DT = LY::DT, CL = LY::CL, SUB = LY::SUB, RS = LY::RS, NP = 16, THREADS = LY::THREADS;
    const int L = p.L;
    if (p.vec) {
        constexpr int VE = 16 / (int)sizeof(T);
        constexpr int CPR = SUB / VE;       // 16-byte chunks per row and sub-stage
        constexpr int RPP = THREADS / CPR;  // rows per pass of the CTA
        static_assert(THREADS % CPR == 0 && DT % RPP == 0, "tile loader mapping");
        const int ch = threadIdx.x % CPR, r0 = threadIdx.x / CPR;
        const int t = part * SUB + ch * VE;  // step within the chunk
        const bool colok = l0 + t < L;
        const T* u = static_cast<const T*>(p.u);
        const T* dl = static_cast<const T*>(p.dl);
        const size_t step = (size_t)RPP * L;
        size_t off = (row0 + r0) * (size_t)L + l0 + t;
#pragma unroll
        for (int it = 0; it < DT / RPP; ++it, off += step) {
            const int r = r0 + it * RPP;
            const bool ok = colok && r < nrows;
            cp_async16(dst + r * RS + t, ok ? u + off : u, ok ? 16 : 0);
            cp_async16(dst + (DT + r) * RS + t, ok ? dl + off : dl, ok ? 16 : 0);
        }
    } else if (part == 0) {
        load_tile<T, NP, DT, CL, RS, THREADS, false, false>(p, dst, row0, 0, nrows, l0);
    }
}

// B (and C) of the whole chunk read with plain 16-byte loads and stored as
// fp32 rows [n][t] of stride FS (zero past the problem).
template <typename T, class CS, bool WITH_C>
__device__ __forceinline__ void load_chunk_bc_f32(const FullParams& p, float* fb, size_t bcrow0, int l0) {
    using LY = ChunkLayout<T, CS>;
    constexpr int CL = LY::CL, FS = LY::FS, NP = 16, THREADS = LY::THREADS;
    const int L = p.L;
    const T* Bs = static_cast<const T*>(p.Bs);
    const T* Cs = static_cast<const T*>(p.Cs);
    if (p.vec) {
        constexpr int VE = 16 / (int)sizeof(T);
        constexpr int CPR = CL / VE;  // 16-byte chunks per row
        constexpr int total = (WITH_C ? 2 : 1) * NP * CPR;
#pragma unroll
        for (int i = threadIdx.x; i < total; i += THREADS) {
            const int r = (i / CPR) % NP, ch = i % CPR, which = i / (NP * CPR);
            const int l = l0 + ch * VE;
            uint4 q = make_uint4(0u, 0u, 0u, 0u);
            if (r < p.N && l < L) q = __ldg(reinterpret_cast<const uint4*>((which ? Cs : Bs) + (bcrow0 + r) * (size_t)L + l));
            float* o = fb + (which * NP + r) * FS + ch * VE;
            if constexpr (LY::F32) {
                *reinterpret_cast<uint4*>(o) = q;
            } else {
                *reinterpret_cast<float4*>(o) = make_float4(__uint_as_float(q.x << 16), __uint_as_float(q.x & 0xffff0000u),
                                                            __uint_as_float(q.y << 16), __uint_as_float(q.y & 0xffff0000u));
                *reinterpret_cast<float4*>(o + 4) = make_float4(__uint_as_float(q.z << 16), __uint_as_float(q.z & 0xffff0000u),
                                                                __uint_as_float(q.w << 16), __uint_as_float(q.w & 0xffff0000u));
            }
        }
    } else {
        constexpr int total = (WITH_C ? 2 : 1) * NP * CL;
        for (int i = threadIdx.x; i < total; i += THREADS) {
            const int r = (i / CL) % NP, t = i % CL, which = i / (NP * CL);
            float v = 0.0f;
            if (r < p.N && l0 + t < L) v = io<T>::ld((which ? Cs : Bs) + (bcrow0 + r) * (size_t)L + l0 + t);
            fb[(which * NP + r) * FS + t] = v;
        }
    }
}

__device__ __forceinline__ void lds4_ordered(const float* p, float (&v)[4]) {
    const unsigned a = (unsigned)__cvta_generic_to_shared(p);
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]) : "r"(a));
}
// The same from a 32-bit shared-window address (a base computed once plus a
// constant offset folds into the load's immediate).
__device__ __forceinline__ void lds4_ordered_u32(unsigned a, float (&v)[4]) {
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]) : "r"(a));
}
__device__ __forceinline__ float ex2_ordered(float x) {
    float y;
    asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float fma_ordered(float a, float b, float c) {
    float y;
    asm volatile("fma.rn.f32 %0, %1, %2, %3;" : "=f"(y) : "f"(a), "f"(b), "f"(c));
    return y;
}
__device__ __forceinline__ float mul_ordered(float a, float b) {
    float y;
    asm volatile("mul.rn.f32 %0, %1, %2;" : "=f"(y) : "f"(a), "f"(b));
    return y;
}

__device__ __forceinline__ void cp_async_wait_upto(int n) {
    switch (n) {
    case 0: cp_async_wait<0>(); break;
    case 1: cp_async_wait<1>(); break;
    case 2: cp_async_wait<2>(); break;
    default: cp_async_wait<3>(); break;
    }
}

template <typename T, class CS, bool PH2>
__global__ void __launch_bounds__(ChunkLayout<T, CS>::THREADS, CS::MINB) full_chunk_kernel(const FullParams p) {
    using LY = ChunkLayout<T, CS>;
    constexpr int G = LY::G, NG = LY::NG, DT = LY::DT, CL = LY::CL, NS = LY::NS, SUB = LY::SUB, RS = LY::RS,
                  FS = LY::FS, NP = 16;
    extern __shared__ __align__(16) unsigned char smem[];
    T* raw = reinterpret_cast<T*>(smem);
    float* sdl = reinterpret_cast<float*>(smem + LY::dl_off);

    // launch 1 (and a single-chunk launch) reads its inputs only after the
    // previous kernel has completed; launch 3 loads its tile before it waits
    // for the carry of launch 2 (the inputs were complete before launch 1 passed
    // its own wait, and launches 1 and 2 signal only after theirs)
    if (!PH2 || p.n_chunks == 1) pdl_wait();
    pdl_launch_dependents();
    const int c = threadIdx.x / G, g = threadIdx.x % G;  // channel within the tile, lane of the channel
    const int tile = blockIdx.x % p.n_tiles;
    const int chunk = blockIdx.x / p.n_tiles;
    const int bk = tile / p.tiles_per_bk;
    const int d0 = (tile % p.tiles_per_bk) * DT;
    const int k = bk % p.K;
    const int d = d0 + c;
    const bool cval = d < p.D;
    const int nrows = min(DT, p.D - d0);
    const size_t row0 = (size_t)bk * p.D + d0;
    const size_t bcrow0 = (size_t)bk * p.N;
    const int l0 = chunk * CL;
    // every sub-stage in flight at once; each is computed as soon as it lands
#pragma unroll
    for (int part = 0; part < NS; ++part) {
        load_chunk_part<T, CS>(p, raw, row0, nrows, l0, part);
        cp_async_commit();
    }
    float* fbc = reinterpret_cast<float*>(smem + LY::bc_off);
    load_chunk_bc_f32<T, CS, PH2>(p, fbc, bcrow0, l0);
    const float bias = cval ? p.bias[(size_t)k * p.D + d] : 0.0f;
    const float dsk = cval ? p.Dskip[(size_t)k * p.D + d] : 0.0f;
    const float* Ad = p.A + ((size_t)k * p.D + d) * p.N;
    float A2r[G == 1 ? 1 : NG];  // G = 2: this lane's A * log2 e
    float* sa2 = reinterpret_cast<float*>(smem + LY::a2_off) + c * NP;  // G = 1: this channel's row (own row only)
    const int sw = (c >> 1) & 3;
    if constexpr (G == 1) {
#pragma unroll
        for (int q = 0; q < NP / 4; ++q) {
            float a[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int n = 4 * q + i;
                a[i] = (cval && n < p.N) ? Ad[n] * kLog2e : 0.0f;
            }
            *reinterpret_cast<float4*>(sa2 + 4 * (q ^ sw)) = make_float4(a[0], a[1], a[2], a[3]);
        }
    } else {
#pragma unroll
        for (int i = 0; i < NG; ++i) {
            const int n = g * NG + i;
            A2r[i] = (cval && n < p.N) ? Ad[n] * kLog2e : 0.0f;
        }
    }
    float h[NG];
#pragma unroll
    for (int i = 0; i < NG; ++i) h[i] = 0.0f;
    constexpr size_t sfl = (size_t)DT * NP;  // floats of one chunk's state (aggP uses the first DT)
    const size_t slot = (size_t)tile * p.n_chunks + chunk;

    const T* ru = raw + c * RS;
    const T* rd = raw + (DT + c) * RS;
    const float* rb = fbc + g * NG * FS;  // this lane's B rows
    const float* rc = rb + NP * FS;
    float* fd = sdl + c * FS;
    const int nvalid = min(CL, p.L - l0);
    T* yrow = static_cast<T*>(p.y) + (row0 + c) * (size_t)p.L + l0;
    float ssum = 0.0f;  // this lane's share of the sum of delta over the chunk
#pragma unroll 1
    for (int part = 0; part < NS; ++part) {
        cp_async_wait_upto(NS - 1 - part);
        __syncthreads();
        // delta = softplus(raw + bias) (Eq. 6) of this channel over the sub-stage,
        // once per element (the G lanes take alternate 4-step groups) with every
        // step independent, as fp32 rows
#pragma unroll
        for (int t0 = part * SUB + 4 * g; t0 < part * SUB + SUB; t0 += 4 * G) {
            float r4[4];
            load4(rd + t0, r4);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float v = r4[j] + bias;
                r4[j] = p.softplus_on ? softplus(v) : v;
                if constexpr (!PH2) ssum += r4[j];  // every step of an aggregated chunk is in range
            }
            *reinterpret_cast<float4*>(fd + t0) = make_float4(r4[0], r4[1], r4[2], r4[3]);
        }
        if constexpr (G > 1) __syncwarp();  // the other lane's delta groups
        if (PH2 && part == 0) {
            pdl_wait();  // the carried-in states of launch 2
            if (chunk > 0) {
                const float4* src = reinterpret_cast<const float4*>(p.incH + (slot - 1) * sfl + (size_t)c * NP + g * NG);
#pragma unroll
                for (int q = 0; q < NG / 4; ++q) {
                    const float4 v = __ldcg(src + q);
                    h[4 * q] = v.x;
                    h[4 * q + 1] = v.y;
                    h[4 * q + 2] = v.z;
                    h[4 * q + 3] = v.w;
                }
            }
        }
#pragma unroll 1
        for (int t0 = part * SUB; t0 < part * SUB + SUB; t0 += 4) {
            float dl4[4], du4[4];
            {
                float u4[4];
                load4(ru + t0, u4);
                load4(fd + t0, dl4);
#pragma unroll
                for (int j = 0; j < 4; ++j) du4[j] = dl4[j] * u4[j];
            }
            const unsigned sb = (unsigned)__cvta_generic_to_shared(rb + t0);  // this lane's B rows at t0
            float ya[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
            for (int q = 0; q < NG / 4; ++q) {
                float a2[4];
                if constexpr (G == 1) {
                    load4(sa2 + 4 * (q ^ sw), a2);
                } else {
#pragma unroll
                    for (int i = 0; i < 4; ++i) a2[i] = A2r[4 * q + i];
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int n = 4 * q + i;  // state index within this lane's share
                    // B, C reads and the exponentials as ordered (volatile) asm: left
                    // free, the compiler hoists all row reads of the block and runs
                    // out of registers
                    float b4[4], c4[4];
                    lds4_ordered_u32(sb + n * FS * 4, b4);
                    if constexpr (PH2) lds4_ordered_u32(sb + (NP + n) * FS * 4, c4);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        h[n] = fmaf(ex2_ordered(dl4[j] * a2[i]), h[n], du4[j] * b4[j]);
                        if constexpr (PH2) ya[j] = fmaf(c4[j], h[n], ya[j]);
                    }
                }
            }
            if constexpr (PH2) {
                if constexpr (G == 1) {
                    float u4[4], o[4];
                    load4(ru + t0, u4);  // read again rather than held across the state loop
#pragma unroll
                    for (int j = 0; j < 4; ++j) o[j] = fmaf(dsk, u4[j], ya[j]);
                    if (cval) store_row<T, 4>(yrow + t0, o, nvalid - t0, p.vec);
                } else {
                    // lane g keeps steps 2g, 2g + 1 and adds the other lane's share
                    const float k0 = g ? ya[2] : ya[0], k1 = g ? ya[3] : ya[1];
                    const float s0 = g ? ya[0] : ya[2], s1 = g ? ya[1] : ya[3];
                    float u4[4], o[2];
                    load4(ru + t0, u4);
                    o[0] = fmaf(dsk, g ? u4[2] : u4[0], k0 + __shfl_xor_sync(0xffffffffu, s0, 1));
                    o[1] = fmaf(dsk, g ? u4[3] : u4[1], k1 + __shfl_xor_sync(0xffffffffu, s1, 1));
                    if (cval) store_row<T, 2>(yrow + t0 + 2 * g, o, nvalid - t0 - 2 * g, p.vec);
                }
            }
        }
    }
    if constexpr (!PH2) {
        if constexpr (G > 1) ssum += __shfl_xor_sync(0xffffffffu, ssum, 1);  // both lanes: lane 0 + lane 1
        if (g == 0) p.aggP[slot * sfl + c] = ssum;
        float4* dst = reinterpret_cast<float4*>(p.aggH + slot * sfl + (size_t)c * NP + g * NG);
#pragma unroll
        for (int q = 0; q < NG / 4; ++q) dst[q] = make_float4(h[4 * q], h[4 * q + 1], h[4 * q + 2], h[4 * q + 3]);
    }
}

// ---------------------------------------------------- streaming variant
// For many channel rows (no L-chunking): the compute structure of the chunked
// kernel over a cp.async ring of TS-step stages.  G lanes per channel (1 or 2)
// own 16 / G states each; per stage the channel's delta row is turned into fp32
// softplus values one stage ahead (the G lanes take alternate 4-step groups of
// their own channel, so no barrier beyond the stage's), B and C are read as fp32
// [n][t] rows four steps per 128-bit broadcast load (bf16 converted
// cooperatively one stage ahead), A * log2 e sits in swizzled shared memory or
// in registers, and the state loop is outermost within a 4-step block.  One
// barrier per stage.
template <int G_, int DT_, int TS_, int MINB_, int V_ = 0, int NSTG_ = 3>
struct StreamShape {
    // V: 0 = A in shared memory, ordered B/C reads and exponentials;
    //    1 = A in registers, ordered reads, exponentials and FMAs; 2 = A in registers, free order
    static constexpr int G = G_, DT = DT_, TS = TS_, MINB = MINB_, V = V_, NSTG = NSTG_;
};

template <typename T, class SS>
struct StreamLayout {
    // TS = 0: one 16-byte chunk per row and stage (4 fp32 or 8 bf16 steps)
    static constexpr int G = SS::G, DT = SS::DT, TS = SS::TS ? SS::TS : 16 / (int)sizeof(T), NP = 16, NSTG = SS::NSTG;
    static constexpr int THREADS = G * DT, NG = NP / G;
    static constexpr bool F32 = sizeof(T) == 4;
    // raw row stride (elements): rows of one 16-byte chunk need no padding (a
    // quarter warp's 128-bit reads of consecutive rows hit distinct banks);
    // longer rows are padded by one chunk
    static constexpr int RS = TS * (int)sizeof(T) == 16 ? TS : TS + 16 / (int)sizeof(T);
    static constexpr int SLOT = (2 * DT + 2 * NP) * RS;  // u, delta, B, C rows of one stage
    static constexpr int FS = F32 ? RS : TS + 4;         // fp32 row stride
    static constexpr size_t raw_bytes = a16((size_t)NSTG * SLOT * sizeof(T));
    // bf16: fp32 delta rows [2][DT][FS] and fp32 B, C rows [2][2 NP][FS] (two
    // slots: the stage being computed and the next); fp32 uses the raw rows
    static constexpr size_t fdl_off = raw_bytes;
    static constexpr size_t fbc_off = fdl_off + (F32 ? 0 : (size_t)2 * DT * FS * 4);
    static constexpr size_t a2_off = fbc_off + (F32 ? 0 : (size_t)2 * 2 * NP * FS * 4);
    static constexpr int V = SS::V;
    static constexpr size_t bytes = a2_off + (V == 0 ? (size_t)DT * NP * 4 : 0);
    static_assert(TS % (4 * G) == 0 && TS * sizeof(T) % 16 == 0 && DT % 32 == 0 && (G == 1 || G == 2) && NSTG >= 3,
                  "stream tile shape");
    static_assert(V != 0 || G == 1, "shared-memory A rows are one lane per channel");
    static_assert(!F32 || RS == FS, "fp32 rows are rewritten in place");
};

template <typename T, class SS>
__global__ void __launch_bounds__(StreamLayout<T, SS>::THREADS, SS::MINB) full_stream_kernel(const FullParams p) {
    pdl_wait();
    pdl_launch_dependents();
    using LY = StreamLayout<T, SS>;
    constexpr int G = LY::G, NG = LY::NG, DT = LY::DT, TS = LY::TS, NP = 16, NSTG = LY::NSTG, RS = LY::RS,
                  SLOT = LY::SLOT, FS = LY::FS, THREADS = LY::THREADS;
    extern __shared__ __align__(16) unsigned char smem[];
    T* raw = reinterpret_cast<T*>(smem);

    const int c = threadIdx.x / G, g = threadIdx.x % G;
    const int tile = blockIdx.x;
    const int bk = tile / p.tiles_per_bk;
    const int d0 = (tile % p.tiles_per_bk) * DT;
    const int k = bk % p.K;
    const int d = d0 + c;
    const bool cval = d < p.D;
    const int nrows = min(DT, p.D - d0);
    const size_t row0 = (size_t)bk * p.D + d0;
    const size_t bcrow0 = (size_t)bk * p.N;
    const int L = p.L;
    const int nst = (L + TS - 1) / TS;
#pragma unroll
    for (int q = 0; q < NSTG - 1; ++q) {
        if (q < nst) load_tile<T, NP, DT, TS, RS, THREADS, true>(p, raw + q * SLOT, row0, bcrow0, nrows, q * TS);
        cp_async_commit();
    }
    const float bias = cval ? p.bias[(size_t)k * p.D + d] : 0.0f;
    const float dsk = cval ? p.Dskip[(size_t)k * p.D + d] : 0.0f;
    const float* Ad = p.A + ((size_t)k * p.D + d) * p.N;
    constexpr int V = LY::V;
    float A2r[V == 0 ? 1 : NG];  // V > 0: this lane's A * log2 e
    float* sa2 = reinterpret_cast<float*>(smem + LY::a2_off) + c * NP;  // V = 0: this channel's row (own row only)
    const int sw = (c >> 1) & 3;
    if constexpr (V == 0) {
#pragma unroll
        for (int q = 0; q < NP / 4; ++q) {
            float a[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int n = 4 * q + i;
                a[i] = (cval && n < p.N) ? Ad[n] * kLog2e : 0.0f;
            }
            *reinterpret_cast<float4*>(sa2 + 4 * (q ^ sw)) = make_float4(a[0], a[1], a[2], a[3]);
        }
    } else {
#pragma unroll
        for (int i = 0; i < NG; ++i) {
            const int n = g * NG + i;
            A2r[i] = (cval && n < p.N) ? Ad[n] * kLog2e : 0.0f;
        }
    }
    float h[NG];
#pragma unroll
    for (int i = 0; i < NG; ++i) h[i] = 0.0f;
    T* yrow = static_cast<T*>(p.y) + (row0 + c) * (size_t)L;

    // fp32 delta row of stage st (this channel) and fp32 B / C rows
    auto fdl_of = [&](int st) -> float* {
        if constexpr (LY::F32) return reinterpret_cast<float*>(raw + (st % NSTG) * SLOT + (DT + c) * RS);
        else return reinterpret_cast<float*>(smem + LY::fdl_off) + ((st & 1) * DT + c) * FS;
    };
    auto fbc_of = [&](int st) -> const float* {
        if constexpr (LY::F32) return reinterpret_cast<const float*>(raw + (st % NSTG) * SLOT + 2 * DT * RS);
        else return reinterpret_cast<const float*>(smem + LY::fbc_off) + (st & 1) * 2 * NP * FS;
    };
    // delta = softplus(raw + bias) (Eq. 6) of this channel over stage st, in fp32
    // (the G lanes take alternate 4-step groups); bf16 storage also converts the
    // stage's B and C rows (cooperatively)
    auto prepare = [&](int st) {
        const T* rd = raw + (st % NSTG) * SLOT + (DT + c) * RS;
        float* fd = fdl_of(st);
#pragma unroll
        for (int t0 = 4 * g; t0 < TS; t0 += 4 * G) {
            float r4[4];
            load4(rd + t0, r4);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float v = r4[j] + bias;
                r4[j] = p.softplus_on ? softplus(v) : v;
            }
            *reinterpret_cast<float4*>(fd + t0) = make_float4(r4[0], r4[1], r4[2], r4[3]);
        }
        if constexpr (!LY::F32) {
            const T* rbc = raw + (st % NSTG) * SLOT + 2 * DT * RS;
            float* fbc = reinterpret_cast<float*>(smem + LY::fbc_off) + (st & 1) * 2 * NP * FS;
            for (int i = threadIdx.x; i < 2 * NP * TS / 4; i += THREADS) {
                const int r = i / (TS / 4), t0 = 4 * (i % (TS / 4));
                float v4[4];
                load4(rbc + r * RS + t0, v4);
                *reinterpret_cast<float4*>(fbc + r * FS + t0) = make_float4(v4[0], v4[1], v4[2], v4[3]);
            }
        }
    };
    cp_async_wait<NSTG - 2>();
    __syncthreads();
    prepare(0);
    for (int s = 0; s < nst; ++s) {
        const int l0 = s * TS;
        const int nvalid = min(TS, L - l0);
        cp_async_wait<NSTG - 3>();  // stages <= s+1 have landed
        __syncthreads();            // ... for every thread; stage s's fp32 rows are prepared
        if (s + NSTG - 1 < nst)
            load_tile<T, NP, DT, TS, RS, THREADS, true>(p, raw + ((s + NSTG - 1) % NSTG) * SLOT, row0, bcrow0,
                                                        nrows, l0 + (NSTG - 1) * TS);
        cp_async_commit();
        if (s + 1 < nst) prepare(s + 1);
        const T* ru = raw + (s % NSTG) * SLOT + c * RS;
        const float* fd = fdl_of(s);
        constexpr int BS = LY::F32 ? RS : FS;  // fp32 B / C row stride
        const float* rb = fbc_of(s) + g * NG * BS;  // this lane's B rows
        const float* rc = rb + NP * BS;
#pragma unroll 1
        for (int t0 = 0; t0 < TS; t0 += 4) {
            float dl4[4], du4[4];
            {
                float u4[4];
                load4(ru + t0, u4);
                load4(fd + t0, dl4);
#pragma unroll
                for (int j = 0; j < 4; ++j) du4[j] = dl4[j] * u4[j];
            }
            const unsigned sb = (unsigned)__cvta_generic_to_shared(rb + t0);  // this lane's B rows at t0
            float ya[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
            for (int q = 0; q < NG / 4; ++q) {
                float a2[4];
                if constexpr (V == 0) {
                    load4(sa2 + 4 * (q ^ sw), a2);
                } else {
#pragma unroll
                    for (int i = 0; i < 4; ++i) a2[i] = A2r[4 * q + i];
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int n = 4 * q + i;
                    float b4[4], c4[4];
                    if constexpr (V == 2) {
                        load4(rb + n * BS + t0, b4);
                        load4(rc + n * BS + t0, c4);
                    } else {
                        // B row n and C row n of this 4-step block: fixed offsets from sb
                        lds4_ordered_u32(sb + n * BS * 4, b4);
                        lds4_ordered_u32(sb + (NP + n) * BS * 4, c4);
                    }
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        if constexpr (V == 0) {
                            h[n] = fmaf(ex2_ordered(dl4[j] * a2[i]), h[n], du4[j] * b4[j]);
                            ya[j] = fmaf(c4[j], h[n], ya[j]);
                        } else if constexpr (V == 1) {
                            h[n] = fma_ordered(ex2_ordered(mul_ordered(dl4[j], a2[i])), h[n], mul_ordered(du4[j], b4[j]));
                            ya[j] = fma_ordered(c4[j], h[n], ya[j]);
                        } else {
                            h[n] = fmaf(ex2(dl4[j] * a2[i]), h[n], du4[j] * b4[j]);
                            ya[j] = fmaf(c4[j], h[n], ya[j]);
                        }
                    }
                }
            }
            float u4[4];
            load4(ru + t0, u4);  // read again rather than held across the state loop
            if constexpr (G == 1) {
                float o[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) o[j] = fmaf(dsk, u4[j], ya[j]);
                if (cval) store_row<T, 4>(yrow + l0 + t0, o, nvalid - t0, p.vec);
            } else {
                // lane g keeps steps 2g, 2g + 1 and adds the other lane's share
                const float k0 = g ? ya[2] : ya[0], k1 = g ? ya[3] : ya[1];
                const float s0 = g ? ya[0] : ya[2], s1 = g ? ya[1] : ya[3];
                float o[2];
                o[0] = fmaf(dsk, g ? u4[2] : u4[0], k0 + __shfl_xor_sync(0xffffffffu, s0, 1));
                o[1] = fmaf(dsk, g ? u4[3] : u4[1], k1 + __shfl_xor_sync(0xffffffffu, s1, 1));
                if (cval) store_row<T, 2>(yrow + l0 + t0 + 2 * g, o, nvalid - t0 - 2 * g, p.vec);
            }
        }
    }
    cp_async_wait<0>();
}

// ---------------------------------------------------- packed streaming variant
// For many channel rows (no L-chunking), with the state update on the packed
// f32x2 operations: G lanes per channel (1, 2 or 4) each own 16 / G states,
// held as pairs (n, n+1).  Per step and pair: Abar = 2^(delta A log2 e) (one
// packed product, two ex2), Bbar u = (delta u) B (one packed product),
// h = Abar h + Bbar u and the output sum C.h (two packed FMAs), so a state
// update costs two FMA-pipe instructions and one ex2 instead of four and one.
// The stage's B and C rows are transposed once per stage into fp32 [t][B..C]
// rows, so a lane reads the pairs of its states at step t as 128-bit
// broadcast loads; delta = softplus(raw + bias) is computed one stage ahead
// on the packed operations as well (the G lanes of a channel split the
// stage's steps).  cp.async ring of 8-step stages, one barrier per stage.
template <int G_, int DT_, int MINB_, int TS_ = 8, int NSTG_ = 3>
struct PackedShape {
    // TS = 0: one 16-byte chunk per row and stage (4 fp32 or 8 bf16 steps)
    static constexpr int G = G_, DT = DT_, MINB = MINB_, TS = TS_, NSTG = NSTG_;
};

template <typename T, class PS>
struct PackedLayout {
    static constexpr int G = PS::G, DT = PS::DT, MINB = PS::MINB, NP = 16, NG = NP / G, NPR = NG / 2;
    static constexpr int TS = PS::TS ? PS::TS : 16 / (int)sizeof(T), NSTG = PS::NSTG;
    static constexpr int THREADS = G * DT;
    static constexpr bool F32 = sizeof(T) == 4;
    // raw row stride (elements): rows of one 16-byte chunk need no padding (a
    // quarter warp's 128-bit reads of consecutive rows hit distinct banks);
    // longer rows are padded by one chunk
    static constexpr int RS = TS * (int)sizeof(T) == 16 ? TS : TS + 16 / (int)sizeof(T);
    static constexpr int SLOT = (2 * DT + 2 * NP) * RS;  // u, delta, B, C rows of one stage
    static constexpr int FS = F32 ? RS : TS + 4;         // fp32 delta row stride
    static constexpr int BCW = 2 * NP;                   // floats per transposed step: B[0..15], C[0..15]
    static constexpr size_t raw_bytes = a16((size_t)NSTG * SLOT * sizeof(T));
    // bf16: fp32 delta rows [2][DT][FS]; fp32 rewrites the raw delta rows in place
    static constexpr size_t fdl_off = raw_bytes;
    static constexpr size_t bct_off = fdl_off + (F32 ? 0 : (size_t)2 * DT * FS * 4);  // fp32 [2][TS][BCW]
    static constexpr size_t bytes = bct_off + (size_t)2 * TS * BCW * 4;
    static_assert((G == 1 || G == 2 || G == 4) && DT % 32 == 0 && THREADS % 32 == 0 && TS % 4 == 0 &&
                      (TS / G) % 2 == 0 && NSTG >= 3, "packed tile shape");
    static_assert(!F32 || RS == FS, "fp32 delta rows are rewritten in place");
};

template <typename T, class PS>
__global__ void __launch_bounds__(PackedLayout<T, PS>::THREADS, PS::MINB) full_packed_kernel(const FullParams p) {
    pdl_wait();
    pdl_launch_dependents();
    using LY = PackedLayout<T, PS>;
    constexpr int G = LY::G, NG = LY::NG, NPR = LY::NPR, DT = LY::DT, TS = LY::TS, NP = 16, NSTG = LY::NSTG,
                  RS = LY::RS, SLOT = LY::SLOT, FS = LY::FS, BCW = LY::BCW, THREADS = LY::THREADS;
    extern __shared__ __align__(16) unsigned char smem[];
    T* raw = reinterpret_cast<T*>(smem);

    const int c = threadIdx.x / G, g = threadIdx.x % G;
    const int tile = blockIdx.x;
    const int bk = tile / p.tiles_per_bk;
    const int d0 = (tile % p.tiles_per_bk) * DT;
    const int k = bk % p.K;
    const int d = d0 + c;
    const bool cval = d < p.D;
    const int nrows = min(DT, p.D - d0);
    const size_t row0 = (size_t)bk * p.D + d0;
    const size_t bcrow0 = (size_t)bk * p.N;
    const int L = p.L;
    const int nst = (L + TS - 1) / TS;
#pragma unroll
    for (int q = 0; q < NSTG - 1; ++q) {
        if (q < nst) load_tile<T, NP, DT, TS, RS, THREADS, true>(p, raw + q * SLOT, row0, bcrow0, nrows, q * TS);
        cp_async_commit();
    }
    const float bias = cval ? p.bias[(size_t)k * p.D + d] : 0.0f;
    const float dsk = cval ? p.Dskip[(size_t)k * p.D + d] : 0.0f;
    const float* Ad = p.A + ((size_t)k * p.D + d) * p.N;
    float2 A2[NPR], h[NPR];
#pragma unroll
    for (int i = 0; i < NPR; ++i) {
        const int n = g * NG + 2 * i;
        A2[i] = make_float2((cval && n < p.N) ? Ad[n] * kLog2e : 0.0f, (cval && n + 1 < p.N) ? Ad[n + 1] * kLog2e : 0.0f);
        h[i] = make_float2(0.0f, 0.0f);
    }
    T* yrow = static_cast<T*>(p.y) + (row0 + c) * (size_t)L;

    auto fdl_of = [&](int st) -> float* {
        if constexpr (LY::F32) return reinterpret_cast<float*>(raw + (st % NSTG) * SLOT + (DT + c) * RS);
        else return reinterpret_cast<float*>(smem + LY::fdl_off) + ((st & 1) * DT + c) * FS;
    };
    auto bct_of = [&](int st) -> float* { return reinterpret_cast<float*>(smem + LY::bct_off) + (st & 1) * TS * BCW; };
    // stage st: delta = softplus(raw + bias) (Eq. 6) of this lane's share of its
    // channel's steps, in fp32; the B and C rows transposed to fp32 [t][B..C]
    auto prepare = [&](int st) {
        constexpr int SPL = TS / G;  // steps per lane
        const T* rd = raw + (st % NSTG) * SLOT + (DT + c) * RS + g * SPL;
        float* fd = fdl_of(st) + g * SPL;
#pragma unroll
        for (int j = 0; j < SPL; j += 2) {
            float2 v = make_float2(io<T>::cvt(rd[j]) + bias, io<T>::cvt(rd[j + 1]) + bias);
            if (p.softplus_on) v = softplus2(v);
            *reinterpret_cast<float2*>(fd + j) = v;
        }
        const T* rb = raw + (st % NSTG) * SLOT + 2 * DT * RS;  // B rows, then C rows, [2 NP][RS]
        float* bo = bct_of(st);
        for (int i = threadIdx.x; i < BCW * TS; i += THREADS) {
            const int r = i % BCW, t = i / BCW;
            bo[t * BCW + r] = io<T>::cvt(rb[r * RS + t]);
        }
    };
    cp_async_wait<NSTG - 2>();
    __syncthreads();
    prepare(0);
    for (int s = 0; s < nst; ++s) {
        const int l0 = s * TS;
        const int nvalid = min(TS, L - l0);
        cp_async_wait<NSTG - 3>();  // stages <= s+1 have landed
        __syncthreads();            // ... for every thread; stage s is prepared
        if (s + NSTG - 1 < nst)
            load_tile<T, NP, DT, TS, RS, THREADS, true>(p, raw + ((s + NSTG - 1) % NSTG) * SLOT, row0, bcrow0, nrows,
                                                        l0 + (NSTG - 1) * TS);
        cp_async_commit();
        if (s + 1 < nst) prepare(s + 1);
        const T* ru = raw + (s % NSTG) * SLOT + c * RS;
        const float* fd = fdl_of(s);
        const float* bct = bct_of(s) + g * NG;  // this lane's B states of step 0 (C at + NP)
#pragma unroll 1
        for (int t0 = 0; t0 < TS; t0 += 4) {
            float u4[4], d4[4];
            load4(ru + t0, u4);
            load4(fd + t0, d4);
            float yp[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 dd = make_float2(d4[j], d4[j]);
                const float du = d4[j] * u4[j];
                const float2 uu = make_float2(du, du);
                const float* bt = bct + (t0 + j) * BCW;
                float2 ya = make_float2(0.0f, 0.0f);
#pragma unroll
                for (int q = 0; q < NG / 4; ++q) {
                    const float4 b = *reinterpret_cast<const float4*>(bt + 4 * q);
                    const float4 cc = *reinterpret_cast<const float4*>(bt + NP + 4 * q);
                    {
                        const float2 x = __fmul2_rn(dd, A2[2 * q]);
                        const float2 a = make_float2(ex2(x.x), ex2(x.y));
                        h[2 * q] = __ffma2_rn(a, h[2 * q], __fmul2_rn(uu, make_float2(b.x, b.y)));
                        ya = __ffma2_rn(make_float2(cc.x, cc.y), h[2 * q], ya);
                    }
                    {
                        const float2 x = __fmul2_rn(dd, A2[2 * q + 1]);
                        const float2 a = make_float2(ex2(x.x), ex2(x.y));
                        h[2 * q + 1] = __ffma2_rn(a, h[2 * q + 1], __fmul2_rn(uu, make_float2(b.z, b.w)));
                        ya = __ffma2_rn(make_float2(cc.z, cc.w), h[2 * q + 1], ya);
                    }
                }
                yp[j] = ya.x + ya.y;
            }
            // y = sum over the channel's lanes + D u, stored straight from registers
            if constexpr (G == 1) {
                float o[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) o[j] = fmaf(dsk, u4[j], yp[j]);
                if (cval) store_row<T, 4>(yrow + l0 + t0, o, nvalid - t0, p.vec);
            } else if constexpr (G == 2) {
                // lane g keeps steps 2g and 2g+1
                const float k0 = g ? yp[2] : yp[0], k1 = g ? yp[3] : yp[1];
                const float s0 = g ? yp[0] : yp[2], s1 = g ? yp[1] : yp[3];
                float o[2];
                o[0] = fmaf(dsk, g ? u4[2] : u4[0], k0 + __shfl_xor_sync(0xffffffffu, s0, 1));
                o[1] = fmaf(dsk, g ? u4[3] : u4[1], k1 + __shfl_xor_sync(0xffffffffu, s1, 1));
                if (cval) store_row<T, 2>(yrow + l0 + t0 + 2 * g, o, nvalid - t0 - 2 * g, p.vec);
            } else {
                const bool hi = g & 2;
                float k0 = hi ? yp[2] : yp[0], k1 = hi ? yp[3] : yp[1];
                const float s0 = hi ? yp[0] : yp[2], s1 = hi ? yp[1] : yp[3];
                k0 += __shfl_xor_sync(0xffffffffu, s0, 2);
                k1 += __shfl_xor_sync(0xffffffffu, s1, 2);
                const bool odd = g & 1;
                const float kk = odd ? k1 : k0, ss = odd ? k0 : k1;
                float o[1];
                o[0] = fmaf(dsk, sel4(u4, g), kk + __shfl_xor_sync(0xffffffffu, ss, 1));
                if (cval) store_row<T, 1>(yrow + l0 + t0 + g, o, nvalid - t0 - g, false);
            }
        }
    }
    cp_async_wait<0>();
}

// ------------------------------------- warp-specialised variant (tensor copies)
// The packed state update of the streaming variant, with the tile movement
// taken off the compute warps.  A CTA is CW consumer warps (one channel per
// lane, all 16 states in registers) and one producer warp.  The producer
// issues, per stage of TS steps, four tiled tensor copies (u and delta:
// DT rows x TS steps, B and C: 16 rows x TS steps) into an NSTG-deep ring
// and, once a stage has landed, converts its B and C rows into fp32
// [t][B0..15, C0..15] rows for broadcast reads.  Stages are handed over with
// mbarriers (landed / ready / released), so no barrier spans the CTA and the
// copies of the next stages overlap the consumers' arithmetic.  Each
// consumer lane computes delta = softplus(raw + bias) of its own row of the
// stage, runs the packed update (the same operations, in the same order, as
// full_packed_kernel: its y is bit-identical) and stores y from registers.
// Requires rows of 16-byte multiples and 16-byte aligned tensors (the host
// picks this variant only then); every wait is bounded.
// Gathering from the map (p.gather_h > 0, App. A cross-scan without the
// cross-scanned sequences): direction k's u rows are the (b, d) planes of x
// (k = 0, 2) or of its transpose xt (k = 1, 3), and the reversed directions
// (k = 2, 3) load the mirrored box, steps [L - (s+1) TS, L - s TS), and read
// it from the end, so each step sees the value the cross-scan would have put
// there (the same operations: y is bit-identical to the scan of xs).
// Low-rank Delta (RP > 0, Eq. 6's s_Delta = Linear_D(Linear_R(u)) with the
// rank-R expansion fused into the scan): the second box of a stage is z
// (16 rows x TS steps, fp32, rows past R zero) instead of the raw Deltas, and
// each consumer lane forms its channel's raw Delta per step as
// sum_r Wup[k,d,r] z_r (r in order, as the selection kernel's epilogue does,
// so fp32 results are bit-identical to selection -> raw Deltas -> scan), with
// its Wup row (RP >= R values, zero-padded) in registers.
template <int CW_, int TS_, int NSTG_, int MINB_, int RP_ = 0, bool GATHER_ = false>
struct WsShape {
    static constexpr int CW = CW_, TS = TS_, NSTG = NSTG_, MINB = MINB_, RP = RP_;
    static constexpr bool GATHER = GATHER_;  // u gathered from the map (see above)
};

struct TensorMaps {
    CUtensorMap u, dl, B, C;  // [B*K][D][L] (u, delta) and [B*K][N][L] (B, C)
    CUtensorMap u2;           // gathering from the map: u is x [B][D][L] and u2 its transpose xt
};

template <typename T, class WS>
struct WsTileLayout {
    static constexpr int CW = WS::CW, DT = 32 * CW, NP = 16, TS = WS::TS, NSTG = WS::NSTG;
    static constexpr int THREADS = DT + 32;
    static constexpr int U_BYTES = DT * TS * (int)sizeof(T);   // one u (or delta) box
    static constexpr int DL_BYTES = WS::RP ? NP * TS * 4 : U_BYTES;  // the delta box, or the z box (fp32)
    static constexpr int BC_BYTES = NP * TS * (int)sizeof(T);  // one B (or C) box
    static constexpr int B_OFF = U_BYTES + DL_BYTES;            // B box within a stage (C follows)
    static constexpr int RAW_STAGE = U_BYTES + DL_BYTES + 2 * BC_BYTES;
    static constexpr int BCT_STAGE = TS * 2 * NP * 4;           // fp32 [TS][B0..15, C0..15]
    static constexpr size_t bct_off = (size_t)NSTG * RAW_STAGE;
    static constexpr size_t wup_off = bct_off + (size_t)NSTG * BCT_STAGE;  // low rank: fp32 [DT][RP + 1] Wup rows
    static constexpr size_t bar_off = wup_off + (WS::RP ? (size_t)DT * (WS::RP + 1) * 4 : 0);
    static constexpr size_t bytes = bar_off + (size_t)3 * NSTG * 8;
    static_assert(U_BYTES % 128 == 0 && BC_BYTES % 128 == 0 && TS % 4 == 0 && TS * sizeof(T) % 16 == 0,
                  "tensor-copy boxes: 16-byte rows, 128-byte aligned boxes");
};

constexpr uint64_t kStageWaitNs = 1000000000ull;  // 1 s per stage hand-over

template <typename T, class WS>
__global__ void __launch_bounds__(WsTileLayout<T, WS>::THREADS, WS::MINB)
    full_ws_kernel(const FullParams p, const __grid_constant__ TensorMaps tm) {
    pdl_wait();
    pdl_launch_dependents();
    using LY = WsTileLayout<T, WS>;
    constexpr int DT = LY::DT, NP = 16, TS = LY::TS, NSTG = LY::NSTG, NPR = NP / 2;
    extern __shared__ __align__(128) unsigned char smem_ws[];
    unsigned char* smem = smem_ws;
    const uint32_t sbase = smem_u32(smem);
    const uint32_t bar0 = sbase + (uint32_t)LY::bar_off;
    // landed[i]: the four copies of the stage in slot i arrived; ready[i]: its
    // B/C rows are converted; released[i]: every consumer warp is done with it
    auto landed = [&](int i) { return bar0 + 8u * i; };
    auto ready = [&](int i) { return bar0 + 8u * (NSTG + i); };
    auto released = [&](int i) { return bar0 + 8u * (2 * NSTG + i); };
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int tile = blockIdx.x;
    const int bk = tile / p.tiles_per_bk;
    const int d0 = (tile % p.tiles_per_bk) * DT;
    const int k = bk % p.K;
    const int L = p.L;
    const int nst = (L + TS - 1) / TS;
    const int cwarps = min(LY::CW, (p.D - d0 + 31) / 32);  // consumer warps with at least one channel
    if (tid == 0) {
        for (int i = 0; i < NSTG; ++i) {
            mbarrier_init(landed(i), 1);
            mbarrier_init(ready(i), 32);
            mbarrier_init(released(i), cwarps);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    __syncthreads();
    if (warp == LY::CW) {
        // ------------------------------------------------------ producer warp
        // u: the rows of (b, k), or gathered from x / xt (see above)
        constexpr bool gather = WS::GATHER;
        const CUtensorMap* um = (gather && (k & 1)) ? &tm.u2 : &tm.u;
        const int uz = gather ? bk / p.K : bk;
        const bool urev = gather && k >= 2;
        int issued = 0;  // stages whose copies have been issued (0 .. issued-1)
        auto issue = [&](int s) {
            issued = s + 1;
            const int slot = s % NSTG;
            const uint32_t dst = sbase + (uint32_t)(slot * LY::RAW_STAGE);
            mbarrier_expect_tx(landed(slot), (unsigned)LY::RAW_STAGE);
            tma_load_3d(dst, um, urev ? L - (s + 1) * TS : s * TS, d0, uz, landed(slot));
            tma_load_3d(dst + LY::U_BYTES, &tm.dl, s * TS, WS::RP ? 0 : d0, bk, landed(slot));
            tma_load_3d(dst + LY::B_OFF, &tm.B, s * TS, 0, bk, landed(slot));
            tma_load_3d(dst + LY::B_OFF + LY::BC_BYTES, &tm.C, s * TS, 0, bk, landed(slot));
        };
        if (lane == 0)
            for (int s = 0; s < NSTG && s < nst; ++s) issue(s);
        issued = __shfl_sync(0xffffffffu, issued, 0);
        int seen = 0;  // stages whose copies this warp has seen land
        bool ok = true;
        // (every wait's outcome is made warp-uniform, so that no lane leaves a
        // loop whose warp-wide operations the others still execute)
        for (int s = 0; s < nst; ++s) {
            const int slot = s % NSTG;
            if (!(ok = __all_sync(0xffffffffu, mbarrier_wait(landed(slot), (s / NSTG) & 1, kStageWaitNs)))) break;
            seen = s + 1;
            // lane r converts row r of [B rows 0..15, C rows 0..15] into column r
            const T* rb = reinterpret_cast<const T*>(smem + slot * LY::RAW_STAGE + LY::B_OFF) + lane * TS;
            float* bo = reinterpret_cast<float*>(smem + LY::bct_off + slot * LY::BCT_STAGE);
#pragma unroll
            for (int t = 0; t < TS; ++t) bo[t * 2 * NP + lane] = io<T>::cvt(rb[t]);
            __syncwarp();
            // (test hook: the first stage is never handed over, so every wait on it runs out)
            if (!(p.suppress && s == 0)) mbarrier_arrive(ready(slot));
            // refill the slot of stage s - 1 once the consumers released it
            if (s >= 1 && s - 1 + NSTG < nst) {
                const int ps = (s - 1) % NSTG;
                if (!(ok = __all_sync(0xffffffffu, mbarrier_wait(released(ps), ((s - 1) / NSTG) & 1, kStageWaitNs))))
                    break;
                if (lane == 0) issue(s - 1 + NSTG);
                issued = __shfl_sync(0xffffffffu, issued, 0);
            }
        }
        if (!ok) {
            if (lane == 0) atomicOr(&p.hdr->err, kErrTimeout);
            // every copy issued must land before the CTA exits
            for (int s = seen; s < issued; ++s) mbarrier_wait(landed(s % NSTG), (s / NSTG) & 1, kStageWaitNs);
        }
        return;
    }
    if (warp >= cwarps) return;  // a tile's channels past D: no work, not counted by `released`
    // -------------------------------------------------------- consumer warps
    const bool urev = WS::GATHER && k >= 2;  // u arrives mirrored (see above)
    const int c = tid;
    const int d = d0 + c;
    const bool cval = d < p.D;
    const size_t row0 = (size_t)bk * p.D + d0;
    const float bias = cval ? p.bias[(size_t)k * p.D + d] : 0.0f;
    const float dsk = cval ? p.Dskip[(size_t)k * p.D + d] : 0.0f;
    const float* Ad = p.A + ((size_t)k * p.D + d) * p.N;
    float2 A2[NPR], h[NPR];
#pragma unroll
    for (int i = 0; i < NPR; ++i) {
        const int n = 2 * i;
        A2[i] = make_float2((cval && n < p.N) ? Ad[n] * kLog2e : 0.0f, (cval && n + 1 < p.N) ? Ad[n + 1] * kLog2e : 0.0f);
        h[i] = make_float2(0.0f, 0.0f);
    }
    T* yrow = static_cast<T*>(p.y) + (row0 + c) * (size_t)L;
    constexpr int RP = WS::RP > 0 ? WS::RP : 1;
    // low rank: this channel's Wup row, in the lane's own shared-memory row (a
    // padded stride: conflict-free) to leave the registers to the states
    float* wr = reinterpret_cast<float*>(smem + LY::wup_off) + c * (RP + 1);
    if constexpr (WS::RP > 0) {
#pragma unroll
        for (int r = 0; r < RP; ++r) wr[r] = (cval && r < p.R) ? p.Wup[((size_t)k * p.D + d) * p.R + r] : 0.0f;
    }
    for (int s = 0; s < nst; ++s) {
        const int slot = s % NSTG;
        if (!__all_sync(0xffffffffu, mbarrier_wait(ready(slot), (s / NSTG) & 1, kStageWaitNs))) {
            if (lane == 0) atomicOr(&p.hdr->err, kErrTimeout);
            return;
        }
        const int l0 = s * TS;
        const int nvalid = min(TS, L - l0);
        const T* ru = reinterpret_cast<const T*>(smem + slot * LY::RAW_STAGE) + c * TS;
        const T* rd = reinterpret_cast<const T*>(smem + slot * LY::RAW_STAGE + LY::U_BYTES) + c * TS;
        float uv[TS], dv[TS];
#pragma unroll
        for (int j = 0; j < TS; j += 4) {
            float q[4], w[4];
            if (urev) {
                // the mirrored box, read from its end
                load4(ru + TS - 4 - j, q);
#pragma unroll
                for (int e = 0; e < 4; ++e) uv[j + e] = q[3 - e];
            } else {
                load4(ru + j, q);
#pragma unroll
                for (int e = 0; e < 4; ++e) uv[j + e] = q[e];
            }
            if constexpr (WS::RP == 0) {
                load4(rd + j, w);
#pragma unroll
                for (int e = 0; e < 4; ++e) dv[j + e] = w[e] + bias;
            }
        }
        if constexpr (WS::RP > 0) {
            // raw Delta = sum_r Wup[r] z_r, r in order (the z rows are broadcast reads)
            const float* zr = reinterpret_cast<const float*>(smem + slot * LY::RAW_STAGE + LY::U_BYTES);
            // (packed: each lane of a pair is the same fused multiply-add as fmaf)
            float2 raw[TS / 2];
#pragma unroll
            for (int j = 0; j < TS / 2; ++j) raw[j] = make_float2(0.0f, 0.0f);
#pragma unroll
            for (int r = 0; r < RP; ++r) {
                if (r < p.R) {
                    const float2 w2 = make_float2(wr[r], wr[r]);
#pragma unroll
                    for (int j = 0; j < TS; j += 4) {
                        const float4 z4 = *reinterpret_cast<const float4*>(zr + r * TS + j);
                        raw[j / 2] = __ffma2_rn(w2, make_float2(z4.x, z4.y), raw[j / 2]);
                        raw[j / 2 + 1] = __ffma2_rn(w2, make_float2(z4.z, z4.w), raw[j / 2 + 1]);
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < TS; j += 2) {
                dv[j] = raw[j / 2].x + bias;
                dv[j + 1] = raw[j / 2].y + bias;
            }
        }
        if (p.softplus_on) {
#pragma unroll
            for (int j = 0; j < TS; j += 2) {
                const float2 v = softplus2(make_float2(dv[j], dv[j + 1]));
                dv[j] = v.x;
                dv[j + 1] = v.y;
            }
        }
        const float* bct = reinterpret_cast<const float*>(smem + LY::bct_off + slot * LY::BCT_STAGE);
#pragma unroll
        for (int t0 = 0; t0 < TS; t0 += 4) {
            float yp[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 dd = make_float2(dv[t0 + j], dv[t0 + j]);
                const float du = dv[t0 + j] * uv[t0 + j];
                const float2 uu = make_float2(du, du);
                const float* bt = bct + (t0 + j) * 2 * NP;
                float2 ya = make_float2(0.0f, 0.0f);
#pragma unroll
                for (int q = 0; q < NP / 4; ++q) {
                    const float4 b = *reinterpret_cast<const float4*>(bt + 4 * q);
                    const float4 cc = *reinterpret_cast<const float4*>(bt + NP + 4 * q);
                    {
                        const float2 x = __fmul2_rn(dd, A2[2 * q]);
                        const float2 a = make_float2(ex2(x.x), ex2(x.y));
                        h[2 * q] = __ffma2_rn(a, h[2 * q], __fmul2_rn(uu, make_float2(b.x, b.y)));
                        ya = __ffma2_rn(make_float2(cc.x, cc.y), h[2 * q], ya);
                    }
                    {
                        const float2 x = __fmul2_rn(dd, A2[2 * q + 1]);
                        const float2 a = make_float2(ex2(x.x), ex2(x.y));
                        h[2 * q + 1] = __ffma2_rn(a, h[2 * q + 1], __fmul2_rn(uu, make_float2(b.z, b.w)));
                        ya = __ffma2_rn(make_float2(cc.z, cc.w), h[2 * q + 1], ya);
                    }
                }
                yp[j] = ya.x + ya.y;
            }
            float o[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) o[j] = fmaf(dsk, uv[t0 + j], yp[j]);
            if (cval) store_row<T, 4>(yrow + l0 + t0, o, nvalid - t0, true);
        }
        __syncwarp();
        if (lane == 0) mbarrier_arrive(released(slot));
    }
}

// Launch 2 of the chunked variant: the inclusive state after every chunk,
// inc_m = 2^(A_n log2 e S_m) inc_{m-1} + H_m from inc_{-1} = 0, for every
// (channel, state) of a tile.  The chain is short in arithmetic but long in
// latency, so it is cut in two levels: warp s of a CTA owns segment s (kSegLen
// consecutive chunks) for 32 (channel, state) pairs, folds it from zero, the
// eight segment results are combined in shared memory (a fixed order, so the
// result is deterministic), and each warp refolds its segment from its
// carry-in, writing inc_m.  Groups of kSegs segments follow one another.
constexpr int kSegLen = 16;
constexpr int kSegs = 8;
constexpr int kCarryThreads = 32 * kSegs;  // 32 pairs (2 channels x 16 states) x kSegs segments

template <int DT>
__global__ void __launch_bounds__(kCarryThreads) full_carry_kernel(const FullParams p) {
    constexpr int groups = DT / 2;
    constexpr size_t sfl = (size_t)DT * 16;
    __shared__ float segP[kSegs][32], segH[kSegs][32];
    // launch 3 may start now: before its own wait it reads only the step inputs
    // (complete since launch 1 passed its wait), as this kernel reads A here
    pdl_launch_dependents();
    const int lane = threadIdx.x & 31, seg = threadIdx.x >> 5;
    const int tile = blockIdx.x / groups;
    const int c = (blockIdx.x % groups) * 2 + (lane >> 4), n = lane & 15;
    const int bk = tile / p.tiles_per_bk;
    const int d = (tile % p.tiles_per_bk) * DT + c;
    const int k = bk % p.K;
    const float A2 = (d < p.D && n < p.N) ? p.A[((size_t)k * p.D + d) * p.N + n] * kLog2e : 0.0f;
    const int M = p.n_chunks - 1;  // aggregates to fold: the last chunk's is never needed
    const size_t base = (size_t)tile * p.n_chunks * sfl;
    pdl_wait();  // the aggregates of launch 1
    float carry = 0.0f;  // inclusive state before the current group
    for (int g0 = 0; g0 < M; g0 += kSegs * kSegLen) {
        const int m0 = g0 + seg * kSegLen;
        const float* sp = p.aggP + base + (size_t)m0 * sfl + c;
        const float* hp = p.aggH + base + (size_t)m0 * sfl + (size_t)c * 16 + n;
        float e[kSegLen], hv[kSegLen];
#pragma unroll
        for (int q = 0; q < kSegLen; ++q) {
            const bool ok = m0 + q < M;
            e[q] = ok ? __ldcg(sp + (size_t)q * sfl) : 0.0f;
            hv[q] = ok ? __ldcg(hp + (size_t)q * sfl) : 0.0f;  // past M: identity (factor 1, H 0)
        }
        float P = 1.0f, Hl = 0.0f;
#pragma unroll
        for (int q = 0; q < kSegLen; ++q) {
            e[q] = ex2(A2 * e[q]);
            Hl = fmaf(e[q], Hl, hv[q]);
            P *= e[q];
        }
        segP[seg][lane] = P;
        segH[seg][lane] = Hl;
        __syncthreads();
        float RH = carry;
        for (int s2 = 0; s2 < seg; ++s2) RH = fmaf(segP[s2][lane], RH, segH[s2][lane]);
        float* ip = p.incH + base + (size_t)m0 * sfl + (size_t)c * 16 + n;
#pragma unroll
        for (int q = 0; q < kSegLen; ++q) {
            RH = fmaf(e[q], RH, hv[q]);
            if (m0 + q < M) ip[(size_t)q * sfl] = RH;
        }
        for (int s2 = 0; s2 < kSegs; ++s2) carry = fmaf(segP[s2][lane], carry, segH[s2][lane]);
        __syncthreads();  // segP / segH are rewritten by the next group
    }
}

// ------------------------------------------------------------------ host side

struct KernelInfo {
    const void* fn;  // the kernel that writes y
    size_t smem;
    int G, DT, threads, ts;
    const void* agg = nullptr;  // chunked variant: the aggregate kernel (launch 1)
    bool tma = false;           // warp-specialised variant: takes the tensor maps of u, delta, B and C
};

template <typename T, int NP, class SH, bool ZOH>
KernelInfo info_for() {
    using LY = Layout<T, NP, SH>;
    const void* fn = reinterpret_cast<const void*>(&full_scan_kernel<T, NP, SH, ZOH>);
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
        attr_err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LY::bytes);
    });
    return {attr_err == cudaSuccess ? fn : nullptr, LY::bytes, LY::G, LY::DT, LY::THREADS, LY::TS};
}

template <typename T, bool ZOH>
KernelInfo lanes_info() {
    using LY = Layout<T, 16, LanesShape>;
    const void* fn = reinterpret_cast<const void*>(&full_scan_lanes_kernel<T, ZOH>);
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
        attr_err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LY::raw_bytes);
    });
    return {attr_err == cudaSuccess ? fn : nullptr, LY::raw_bytes, 16, LY::DT, 256, LY::TS};
}

template <typename T, class CS>
KernelInfo chunk_info() {
    using LY = ChunkLayout<T, CS>;
    const void* fa = reinterpret_cast<const void*>(&full_chunk_kernel<T, CS, false>);
    const void* ff = reinterpret_cast<const void*>(&full_chunk_kernel<T, CS, true>);
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
        attr_err = cudaFuncSetAttribute(fa, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LY::bytes);
        if (attr_err == cudaSuccess)
            attr_err = cudaFuncSetAttribute(ff, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LY::bytes);
    });
    const bool ok = attr_err == cudaSuccess;
    return {ok ? ff : nullptr, LY::bytes, LY::G, LY::DT, LY::THREADS, LY::CL, ok ? fa : nullptr};
}

template <typename T, class SS>
KernelInfo stream_info() {
    using LY = StreamLayout<T, SS>;
    const void* fn = reinterpret_cast<const void*>(&full_stream_kernel<T, SS>);
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
        attr_err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LY::bytes);
    });
    return {attr_err == cudaSuccess ? fn : nullptr, LY::bytes, LY::G, LY::DT, LY::THREADS, LY::TS};
}

template <typename T, class PS>
KernelInfo packed_info() {
    using LY = PackedLayout<T, PS>;
    const void* fn = reinterpret_cast<const void*>(&full_packed_kernel<T, PS>);
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
        attr_err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LY::bytes);
    });
    return {attr_err == cudaSuccess ? fn : nullptr, LY::bytes, LY::G, LY::DT, LY::THREADS, LY::TS};
}

template <typename T, class WS>
KernelInfo ws_info() {
    using LY = WsTileLayout<T, WS>;
    const void* fn = reinterpret_cast<const void*>(&full_ws_kernel<T, WS>);
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
        attr_err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LY::bytes);
    });
    KernelInfo ki{attr_err == cudaSuccess ? fn : nullptr, LY::bytes, 1, LY::DT, LY::THREADS, LY::TS};
    ki.tma = true;
    return ki;
}

// The gathering instance of the warp-specialised kernel (u from the map).
KernelInfo ws_gather_info(vmb_dtype dt) {
    return dt == VMB_BF16 ? ws_info<__nv_bfloat16, WsShape<4, 8, 4, 4, 0, true>>()
                          : ws_info<float, WsShape<4, 8, 4, 4, 0, true>>();
}

// The low-rank-Delta instance of the warp-specialised kernel for rank <= RP.
KernelInfo ws_lowrank_info(vmb_dtype dt, int R) {
    if (dt == VMB_BF16)
        return R <= 8 ? ws_info<__nv_bfloat16, WsShape<4, 8, 4, 4, 8>>() : ws_info<__nv_bfloat16, WsShape<4, 8, 4, 4, 16>>();
    return R <= 8 ? ws_info<float, WsShape<4, 8, 4, 4, 8>>() : ws_info<float, WsShape<4, 8, 4, 4, 16>>();
}

// The driver's tensor-map encoder, looked up once (null when unavailable).
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    });
    return fn;
}

// Tensor map of `planes` row-major [rows][L] slabs of u, delta, B or C, read
// in boxes of box_rows rows x box_ts steps (rows past `rows` and steps past L
// read as zero).
bool encode_rows(CUtensorMap* m, const void* base, vmb_dtype dt, int L, int rows, long long planes, int box_ts,
                 int box_rows) {
    const PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (!enc) return false;
    const cuuint64_t es = dt == VMB_BF16 ? 2 : 4;
    const cuuint64_t dims[3] = {(cuuint64_t)L, (cuuint64_t)rows, (cuuint64_t)planes};
    const cuuint64_t strides[2] = {(cuuint64_t)L * es, (cuuint64_t)rows * L * es};
    const cuuint32_t box[3] = {(cuuint32_t)box_ts, (cuuint32_t)box_rows, 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, dt == VMB_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3,
               const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tile shapes per padded state count, in order of preference (fewest lanes
// per channel first).  The zero-order-hold variant uses the first shape.
int shape_count(int np) { return np <= 4 ? 1 : np == 8 ? 2 : 20; }
constexpr int kLanesShape = 7;   // index of the lane-per-state variant (N <= 16 padded to 16)
constexpr int kChunkShape = 8;   // first index of the three-launch chunked variant (shapes 8 to 11)
bool is_chunk_shape(int np, int shape) { return np == 16 && shape >= kChunkShape && shape < kChunkShape + 4; }
constexpr int kStreamShape = 12;  // first index of the streaming one-lane variant (shapes 12 to 15)
bool is_stream_shape(int np, int shape) { return np == 16 && shape >= kStreamShape && shape < kStreamShape + 4; }
constexpr int kPackedShape = 16;  // first index of the packed streaming variant (shapes 16 to 18: G = 1, 2, 4)
bool is_packed_shape(int np, int shape) { return np == 16 && shape >= kPackedShape && shape < kPackedShape + 3; }
constexpr int kWsShape = 19;  // the warp-specialised variant (tensor copies; 16-byte rows and aligned tensors)
bool is_ws_shape(int np, int shape) { return np == 16 && shape == kWsShape; }

template <typename T, bool ZOH>
KernelInfo pick_t(int np, int shape) {
    if (ZOH) shape = 0;
    switch (np) {
    case 1: return info_for<T, 1, Shape<1, 128, 16, 3>, ZOH>();
    case 2: return info_for<T, 2, Shape<1, 128, 16, 3>, ZOH>();
    case 4: return info_for<T, 4, Shape<1, 128, 16, 3>, ZOH>();
    case 8:
        if (shape == 1) return info_for<T, 8, Shape<2, 64, 16, 3>, false>();
        return info_for<T, 8, Shape<1, 128, 8, 3>, ZOH>();
    default:
        switch (shape) {
        case 1: return info_for<T, 16, Shape<2, 128, 8, 3>, false>();
        case 2: return info_for<T, 16, Shape<2, 64, 16, 3>, false>();
        case 3: return info_for<T, 16, Shape<4, 64, 16, 3>, false>();
        case 4: return info_for<T, 16, Shape<4, 32, 32, 3>, false>();
        case 5: return info_for<T, 16, Shape<1, 64, 16, 3>, false>();
        case 6: return info_for<T, 16, Shape<1, 32, 16, 3>, false>();
        case 7: return lanes_info<T, false>();
        case 8: return chunk_info<T, ChunkShape<1, 64, 32, 2, 8>>();
        case 9: return chunk_info<T, ChunkShape<2, 64, 32, 2, 4>>();
        case 10: return chunk_info<T, ChunkShape<1, 64, 64, 4, 5>>();
        case 11: return chunk_info<T, ChunkShape<2, 64, 64, 4, 4>>();
        case 12: return stream_info<T, StreamShape<1, 128, 8, 4, 0>>();
        case 13: return stream_info<T, StreamShape<1, 64, 8, 8, 0>>();
        case 14: return stream_info<T, StreamShape<1, 128, 8, 4, 2>>();
        case 15: return stream_info<T, StreamShape<2, 64, 8, 6, 2>>();
        case 16: return packed_info<T, PackedShape<1, 128, 5, 8, 3>>();
        case 17: return packed_info<T, PackedShape<2, 64, 5, 8, 3>>();
        case 18: return packed_info<T, PackedShape<4, 32, 5, 8, 3>>();
        case 19: return ws_info<T, WsShape<4, 8, 4, 4>>();
        default: return info_for<T, 16, Shape<1, 128, 0, 3, 7>, ZOH>();
        }
    }
}

KernelInfo pick(vmb_dtype dt, int np, int shape, bool zoh) {
    if (dt == VMB_BF16) return zoh ? pick_t<__nv_bfloat16, true>(np, shape) : pick_t<__nv_bfloat16, false>(np, shape);
    return zoh ? pick_t<float, true>(np, shape) : pick_t<float, false>(np, shape);
}

int pad_states(int N) {
    int np = 1;
    while (np < N) np <<= 1;
    return np;
}

// Test-only override of the tile shape and chunk count (vmb_testing.h).
bool forced_plan(int* shape, int* chunks) {
    *shape = forced_full_shape(chunks);
    return *shape >= 0;
}

}  // namespace

// Roles of the tile shapes of one padded state count: "wide" (one lane per
// channel, 128 channels: cheapest per state update), "mid" (two lanes per
// channel), and for sequences that must be cut into chunks "chunk_narrow"
// (one lane per channel, 64 channels) and "chunk_wide" (widest split).
struct ShapeRoles {
    int wide, mid, chunk_narrow, chunk_wide;
};
ShapeRoles roles(int np) {
    if (np >= 16) return {0, 2, 5, 3};
    if (np == 8) return {0, 1, 0, 1};
    return {0, 0, 0, 0};
}

vmb_status plan_full(const ScanArgs& a, ScanPlan* plan) {
    if (a.N < 1 || a.N > 16) return VMB_ERR_UNSUPPORTED;
    const int np = pad_states(a.N);
    const bool zoh = (a.flags & VMB_FLAG_B_ZOH) != 0;
    const long long rows = (long long)a.B * a.K * a.D;
    const int sms = device_sm_count();
    auto info = [&](int sh, KernelInfo* ki, long long* resident) -> vmb_status {
        *ki = pick(a.dtype, np, sh, zoh);
        if (!ki->fn) return VMB_ERR_CUDA;
        int per_sm = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ki->fn, ki->threads, ki->smem) != cudaSuccess)
            return VMB_ERR_CUDA;
        *resident = (long long)(per_sm < 1 ? 1 : per_sm) * sms;
        return VMB_OK;
    };
    // Rules measured on GB300 over the benchmark workloads: 16 states, L >= 128 and
    // at least 128 channel rows per SM -> the warp-specialised kernel when the tensors
    // allow tensor copies, else (at least 256 rows per SM) the packed streaming kernel; otherwise plenty of
    // rows -> one lane per channel; a fair number -> two lanes; too few -> cut L into
    // chunks: the three-launch variant (two lanes per channel, 32-step chunks)
    // while a grid of 64-step one-lane chunks would fit in two waves, else
    // look-back chunks with one lane per channel when they stay long (>= 256
    // steps) and the widest split otherwise (>= 128 steps).
    // the warp-specialised variant needs 16-byte rows and 16-byte aligned
    // tensors (tiled tensor copies) and the driver's tensor-map encoder
    const size_t es = a.dtype == VMB_BF16 ? 2 : 4;
    const auto al16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    const bool tma_ok = np == 16 && (size_t)a.L * es % 16 == 0 && al16(a.u) && al16(a.delta) && al16(a.Bs) &&
                        al16(a.Cs) && al16(a.y) && (a.gather_h == 0 || al16(a.u_t)) &&
                        tensor_map_encoder() != nullptr;
    int shape = 0, n_chunks = 1, forced_chunks = 0, forced_shape = 0;
    KernelInfo ki{};
    long long res = 0;
    vmb_status st;
    if (!zoh && forced_plan(&forced_shape, &forced_chunks)) {
        shape = forced_shape % shape_count(np);
        if (is_ws_shape(np, shape) && !tma_ok) shape = kPackedShape;
        if ((st = info(shape, &ki, &res)) != VMB_OK) return st;
        n_chunks = forced_chunks > 1 ? forced_chunks : 1;
    } else if (zoh) {
        if ((st = info(0, &ki, &res)) != VMB_OK) return st;
        const long long tiles = a.B * a.K * (long long)((a.D + ki.DT - 1) / ki.DT);
        if (rows * 4 < res * ki.threads * 3 && tiles < res) {
            const long long want = (res + tiles - 1) / tiles, mx = (a.L + 255) / 256;
            n_chunks = (int)(want < mx ? want : mx);
        }
    } else if (tma_ok && rows >= 128LL * sms && a.L >= 128) {
        // a fair number of rows and tensors the tensor copies can read: the
        // warp-specialised kernel, one pass over L (measured on GB300: fastest
        // from the batch-32 56x56 map, under a third of a wave of its tiles, up)
        shape = kWsShape;
        if ((st = info(shape, &ki, &res)) != VMB_OK) return st;
    } else if (np == 16 && rows >= 256LL * sms && a.L >= 128) {
        // many rows: the packed streaming one-lane kernel, one pass over L (on
        // very short sequences its stage prologue does not pay off)
        shape = kPackedShape;
        if ((st = info(shape, &ki, &res)) != VMB_OK) return st;
    } else {
        const ShapeRoles r = roles(np);
        if ((st = info(r.wide, &ki, &res)) != VMB_OK) return st;
        shape = r.wide;
        KernelInfo kl{};
        long long rl = 0;
        if (np == 16 && a.L <= 1024 && rows * 4 < res * ki.threads * 3) {
            // short sequences with few rows: one lane per state, single pass
            if ((st = info(kLanesShape, &kl, &rl)) != VMB_OK) return st;
            if (rows * 16 <= rl * kl.threads) {
                shape = kLanesShape;
                ki = kl;
                res = rl;
            }
        }
        if (shape != kLanesShape && rows * 4 < res * ki.threads * 3) {
            KernelInfo km{};
            long long rm = 0;
            if ((st = info(r.mid, &km, &rm)) != VMB_OK) return st;
            KernelInfo kc{}, k9{};
            long long rc = 0, r9 = 0;
            long long chunk_ctas = 0;
            if (np == 16) {
                // few rows: the three-launch chunked variant while a grid of
                // 64-step, one-lane chunks would fit in two waves (beyond that
                // its aggregate traffic outweighs the look-back's second pass).
                // It then runs as two lanes per channel over 32-step chunks,
                // which measured fastest on GB300 with the launches chained
                // (stage-1 maps at batch 1 to 3: 5 to 6% shorter steps than
                // the 64-step chunks)
                if ((st = info(kChunkShape + 2, &kc, &rc)) != VMB_OK) return st;
                if ((st = info(kChunkShape + 1, &k9, &r9)) != VMB_OK) return st;
                chunk_ctas = a.B * a.K * (long long)((a.D + kc.DT - 1) / kc.DT) * ((a.L + kc.ts - 1) / kc.ts);
            }
            if (rows * km.G * 2 >= rm * km.threads) {
                shape = r.mid;
                ki = km;
                res = rm;
            } else if (np == 16 && chunk_ctas <= 2 * rc) {
                shape = kChunkShape + 1;
                ki = k9;
                res = r9;
            } else {
                KernelInfo kn{};
                long long rn = 0;
                if ((st = info(r.chunk_narrow, &kn, &rn)) != VMB_OK) return st;
                const long long tiles_n = a.B * a.K * (long long)((a.D + kn.DT - 1) / kn.DT);
                const long long want_n = (2 * rn + tiles_n - 1) / tiles_n;
                if (a.L / want_n >= 256) {
                    shape = r.chunk_narrow;
                    ki = kn;
                    n_chunks = (int)want_n;
                } else {
                    KernelInfo kw{};
                    long long rw = 0;
                    if ((st = info(r.chunk_wide, &kw, &rw)) != VMB_OK) return st;
                    const long long tiles_w = a.B * a.K * (long long)((a.D + kw.DT - 1) / kw.DT);
                    const long long want_w = (rw + tiles_w - 1) / tiles_w, mx = (a.L + 127) / 128;
                    shape = r.chunk_wide;
                    ki = kw;
                    n_chunks = (int)(want_w < mx ? want_w : mx);
                }
            }
        }
    }
    if (is_chunk_shape(np, shape)) n_chunks = (a.L + ki.ts - 1) / ki.ts;  // chunks of exactly ts steps
    if (is_stream_shape(np, shape) || is_packed_shape(np, shape) || is_ws_shape(np, shape))
        n_chunks = 1;  // one pass over L
    if (n_chunks < 1) n_chunks = 1;
    ScanPlan p{};
    p.np = np;
    p.split = shape;
    p.tile_rows = ki.DT;
    p.tiles_per_bk = (a.D + ki.DT - 1) / ki.DT;
    p.n_seq = a.B * a.K * p.tiles_per_bk;
    int chunk_len = (a.L + n_chunks - 1) / n_chunks;
    chunk_len = (chunk_len + ki.ts - 1) / ki.ts * ki.ts;
    p.n_chunks = (a.L + chunk_len - 1) / chunk_len;
    p.chunk_len = chunk_len;
    p.state_floats = (size_t)ki.DT * np;
    p.ws_bytes = ws_layout(p).total;
    // the warp-specialised kernel's CTAs each stream a whole sequence: a grid of
    // less than one wave launched early would be placed on the SMs that the
    // previous kernel frees first, up to the per-SM limit, and leave the others
    // idle for its whole life (measured on GB300, batch-32 56x56 map after the
    // map transpose: 514 us alone, about 900 us launched early); from a full
    // wave up the early launch is about 3% faster (batch-128 map)
    if (is_ws_shape(np, shape)) p.early = (long long)p.n_seq * p.n_chunks >= res;
    *plan = p;
    return VMB_OK;
}

bool full_plan_gathers(const ScanPlan& plan) { return is_ws_shape(plan.np, plan.split); }

// Raw Deltas of the low-rank form written out (for plans whose kernels read
// materialised Deltas): out[b,k,d,l] = sum_r Wup[k,d,r] z[b,k,r,l], r in order
// (the selection kernel's epilogue order), rounded to the storage type.
template <typename T>
__global__ void __launch_bounds__(256) lowrank_expand_kernel(const float* __restrict__ z, const float* __restrict__ Wup,
                                                             T* __restrict__ out, int K, int D, int R, int L,
                                                             long long total) {
    pdl_wait();
    pdl_launch_dependents();
    for (long long i = blockIdx.x * 256LL + threadIdx.x; i < total; i += (long long)gridDim.x * 256) {
        const int l = (int)(i % L);
        const long long rowi = i / L;  // (b, k, d)
        const int d = (int)(rowi % D);
        const long long bk = rowi / D;
        const int k = (int)(bk % K);
        const float* w = Wup + ((size_t)k * D + d) * R;
        const float* zz = z + (size_t)bk * R * L + l;
        float s = 0.0f;
        for (int r = 0; r < R; ++r) s = fmaf(__ldg(w + r), __ldg(zz + (size_t)r * L), s);
        out[i] = io<T>::to(s);
    }
}

vmb_status launch_lowrank_expand(const float* z, const float* Wup, void* out, int B, int K, int D, int R, int L,
                                 vmb_dtype dt, cudaStream_t stream) {
    long long total = (long long)B * K * D * L;
    int K_ = K, D_ = D, R_ = R, L_ = L;
    const long long want = (total + 255) / 256;
    const unsigned grid = (unsigned)(want < 152LL * 64 ? want : 152LL * 64);
    void* args[] = {(void*)&z, (void*)&Wup, &out, &K_, &D_, &R_, &L_, &total};
    const void* fn = dt == VMB_BF16 ? reinterpret_cast<const void*>(&lowrank_expand_kernel<__nv_bfloat16>)
                                    : reinterpret_cast<const void*>(&lowrank_expand_kernel<float>);
    return launch_kernel(fn, dim3(grid), dim3(256), 0, args, stream) == cudaSuccess ? VMB_OK : VMB_ERR_CUDA;
}

int full_plan_launches(const ScanPlan& plan) {
    return (is_chunk_shape(plan.np, plan.split) && plan.n_chunks > 1) ? 3 : 1;
}

vmb_status launch_full(const ScanArgs& a, const ScanPlan& plan, cudaStream_t stream) {
    const bool lowrank = a.R > 0;
    if ((lowrank || a.gather_h > 0) && !is_ws_shape(plan.np, plan.split)) return VMB_ERR_UNSUPPORTED;
    if (lowrank && a.gather_h > 0) return VMB_ERR_UNSUPPORTED;
    KernelInfo ki = lowrank ? ws_lowrank_info(a.dtype, a.R)
                    : a.gather_h > 0 ? ws_gather_info(a.dtype)
                                     : pick(a.dtype, plan.np, plan.split, (a.flags & VMB_FLAG_B_ZOH) != 0);
    if (!ki.fn) return VMB_ERR_CUDA;
    const size_t es = a.dtype == VMB_BF16 ? 2 : 4;
    FullParams p{};
    p.u = a.u;
    p.dl = a.delta;
    p.A = a.A;
    p.Bs = a.Bs;
    p.Cs = a.Cs;
    p.Dskip = a.Dskip;
    p.bias = a.bias;
    p.y = a.y;
    p.K = a.K;
    p.D = a.D;
    p.N = a.N;
    p.L = a.L;
    p.softplus_on = (a.flags & VMB_FLAG_SOFTPLUS) ? 1 : 0;
    p.tiles_per_bk = plan.tiles_per_bk;
    p.n_tiles = plan.n_seq;
    p.n_chunks = plan.n_chunks;
    p.chunk_len = plan.chunk_len;
    const auto al16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    p.vec = ((size_t)a.L * es % 16 == 0) && al16(a.u) && al16(a.delta) && al16(a.Bs) && al16(a.Cs) && al16(a.y);
    p.suppress = (a.flags & VMB_FLAG_TEST_SUPPRESS_PUBLISH) ? 1 : 0;
    p.gather_h = a.gather_h;
    if (a.gather_h > 0 && !ki.tma) return VMB_ERR_UNSUPPORTED;  // only the warp-specialised kernel gathers
    p.Wup = a.Wup;
    p.R = a.R;
    const WsLayout w = ws_layout(plan);
    unsigned char* ws = static_cast<unsigned char*>(a.ws);
    p.hdr = reinterpret_cast<WsHeader*>(ws);
    p.flags = reinterpret_cast<unsigned*>(ws + w.flags_off);
    p.aggP = reinterpret_cast<float*>(ws + w.aggP_off);
    p.aggH = reinterpret_cast<float*>(ws + w.aggH_off);
    p.incH = reinterpret_cast<float*>(ws + w.incH_off);
    const unsigned grid = (unsigned)(plan.n_seq * plan.n_chunks);
    void* args[] = {&p};
    if (is_chunk_shape(plan.np, plan.split) && plan.n_chunks > 1) {
        // launches 1 and 2 of the chunked variant: aggregates, then the carry fold
        if (!ki.agg) return VMB_ERR_CUDA;
        const unsigned grid_agg = (unsigned)(plan.n_seq * (plan.n_chunks - 1));
        if (launch_kernel(ki.agg, dim3(grid_agg), dim3(ki.threads), ki.smem, args, stream) != cudaSuccess)
            return VMB_ERR_CUDA;
        const unsigned grid_carry = (unsigned)(plan.n_seq * (ki.DT / 2));
        const void* carry = ki.DT == 128 ? reinterpret_cast<const void*>(&full_carry_kernel<128>)
                                         : reinterpret_cast<const void*>(&full_carry_kernel<64>);
        if (launch_kernel(carry, dim3(grid_carry), dim3(kCarryThreads), 0, args, stream) != cudaSuccess)
            return VMB_ERR_CUDA;
        // launch 3 loads its tile and applies the softplus before it waits for the carry
        return launch_kernel(ki.fn, dim3(grid), dim3(ki.threads), ki.smem, args, stream) == cudaSuccess ? VMB_OK
                                                                                                       : VMB_ERR_CUDA;
    }
    if (ki.tma) {
        TensorMaps tm;
        const long long planes = (long long)a.B * a.K;
        const bool gather = a.gather_h > 0;
        // gathering: u and u2 are the map x and its transpose, [B][D][L] each
        bool ok = gather ? encode_rows(&tm.u, a.u, a.dtype, a.L, a.D, a.B, ki.ts, ki.DT) &&
                               encode_rows(&tm.u2, a.u_t, a.dtype, a.L, a.D, a.B, ki.ts, ki.DT)
                         : encode_rows(&tm.u, a.u, a.dtype, a.L, a.D, planes, ki.ts, ki.DT);
        if (!gather) tm.u2 = tm.u;
        // the delta box: DT rows of raw Deltas, or (low rank) the 16 rows of z, fp32
        ok = ok && (lowrank ? encode_rows(&tm.dl, a.delta, VMB_F32, a.L, a.R, planes, ki.ts, 16)
                            : encode_rows(&tm.dl, a.delta, a.dtype, a.L, a.D, planes, ki.ts, ki.DT));
        if (ok &&
            encode_rows(&tm.B, a.Bs, a.dtype, a.L, a.N, planes, ki.ts, 16) &&
            encode_rows(&tm.C, a.Cs, a.dtype, a.L, a.N, planes, ki.ts, 16)) {
            void* targs[] = {&p, &tm};
            return launch_kernel(ki.fn, dim3(grid), dim3(ki.threads), ki.smem, targs, stream, plan.early) ==
                           cudaSuccess
                       ? VMB_OK
                       : VMB_ERR_CUDA;
        }
        // the encoder refused the tensors: the packed streaming variant (same tiles, same
        // results), which reads materialised sequences only
        if (gather || lowrank) return VMB_ERR_UNSUPPORTED;
        ki = pick(a.dtype, plan.np, kPackedShape, false);
        if (!ki.fn) return VMB_ERR_CUDA;
    }
    return launch_kernel(ki.fn, dim3(grid), dim3(ki.threads), ki.smem, args, stream) == cudaSuccess ? VMB_OK
                                                                                                   : VMB_ERR_CUDA;
}

}  // namespace vmb
