// cross_scan_merge.cu - SS2D cross-scan and cross-merge (App. A, "VMamba") for sm_103a.
//
// cross-scan: x[B,D,H,W] -> xs[B,4,D,L].  A CTA stages ppc whole maps (planes)
// in shared memory with a padded row stride, then writes the four direction
// rows of every plane: 0 row-major, 1 column-major, 2 and 3 the reverses of 0
// and 1.  Global loads and stores are 16-byte vectors when rows are 16-byte
// aligned; the padding keeps the column-major reads free of bank conflicts.
//
// Maps of 1024 pixels or more use band kernels instead: one CTA per band of
// rows of one map (eight for the scan, up to 32 for the merge; see below),
// which keeps batch-1 problems parallel.
//
// cross-merge: ys[B,4,D,L] -> out[B,D,H,W], out = (ys0[p0] + ys2[p2]) +
// (ys1[p1] + ys3[p3]) in fp32 in that order.  Directions 0 and 2 are read
// straight from global memory in output order (2 reversed); directions 1 and
// 3 are staged in shared memory keyed by (w, h) so the transposed reads are
// conflict-free.
//
// Index arithmetic uses division by invariant integers via multiply-high
// (Granlund & Montgomery, "Division by invariant integers using
// multiplication", PLDI 1994, round-up variant), valid for dividends < 2^31.
#include "vmb_common.cuh"
#include "vmb_internal.h"

namespace vmb {
namespace {

constexpr int kThreads = 256;
constexpr size_t kMaxSmem = 200 * 1024;

struct FastDiv {
    unsigned d, m, s;
};
FastDiv make_fastdiv(unsigned d) {
    unsigned s = 0;
    while ((1ull << s) < d) ++s;
    const unsigned long long m = ((1ull << 32) * ((1ull << s) - d)) / d + 1;
    return {d, (unsigned)m, s};
}
__device__ __forceinline__ unsigned fdiv(unsigned n, FastDiv f) { return (__umulhi(n, f.m) + n) >> f.s; }

struct CsmParams {
    const void* in;
    void* out;
    int D, H, W, L;
    long long planes;  // B * D
    int ppc;           // planes per CTA
    int vec;
    FastDiv fL, fW, fH, fD;
};

template <typename T>
union Vec {
    uint4 v;
    T e[16 / sizeof(T)];
};

template <typename T>
__global__ void __launch_bounds__(kThreads) cross_scan_kernel(const CsmParams p) {
    pdl_wait();
    pdl_launch_dependents();
    extern __shared__ __align__(16) unsigned char smem_raw[];
    T* sp = reinterpret_cast<T*>(smem_raw);  // [ppc][H][W+1]
    constexpr int VE = 16 / sizeof(T);
    const T* x = static_cast<const T*>(p.in);
    T* xs = static_cast<T*>(p.out);
    const int L = p.L, W = p.W, H = p.H, WP = p.W + 1;
    const long long p0 = (long long)blockIdx.x * p.ppc;
    const int np = (int)min((long long)p.ppc, p.planes - p0);
    const unsigned n = (unsigned)(np * L);
    const T* src = x + p0 * L;
    // stage the planes
    if (p.vec) {
        for (unsigned i = threadIdx.x * VE; i < n; i += kThreads * VE) {
            Vec<T> v;
            v.v = *reinterpret_cast<const uint4*>(src + i);
#pragma unroll
            for (int q = 0; q < VE; ++q) {
                const unsigned e = i + q;
                const unsigned j = fdiv(e, p.fL), r = e - j * L;
                const unsigned h = fdiv(r, p.fW), w = r - h * W;
                sp[(j * H + h) * WP + w] = v.e[q];
            }
        }
    } else {
        for (unsigned e = threadIdx.x; e < n; e += kThreads) {
            const unsigned j = fdiv(e, p.fL), r = e - j * L;
            const unsigned h = fdiv(r, p.fW), w = r - h * W;
            sp[(j * H + h) * WP + w] = src[e];
        }
    }
    __syncthreads();
    // write the four direction rows of every staged plane
#pragma unroll 1
    for (int kd = 0; kd < 4; ++kd) {
        const bool rev = kd >= 2, colmajor = kd & 1;
        if (p.vec) {
            for (unsigned i = threadIdx.x * VE; i < n; i += kThreads * VE) {
                const unsigned j = fdiv(i, p.fL), l = i - j * L;
                const long long pi = p0 + j;
                const unsigned b = fdiv((unsigned)pi, p.fD), d = (unsigned)pi - b * p.D;
                Vec<T> v;
#pragma unroll
                for (int q = 0; q < VE; ++q) {
                    const unsigned m = rev ? L - 1 - (l + q) : l + q;
                    unsigned h, w;
                    if (colmajor) {
                        w = fdiv(m, p.fH);
                        h = m - w * H;
                    } else {
                        h = fdiv(m, p.fW);
                        w = m - h * W;
                    }
                    v.e[q] = sp[(j * H + h) * WP + w];
                }
                *reinterpret_cast<uint4*>(xs + (((long long)b * 4 + kd) * p.D + d) * L + l) = v.v;
            }
        } else {
            for (unsigned i = threadIdx.x; i < n; i += kThreads) {
                const unsigned j = fdiv(i, p.fL), l = i - j * L;
                const long long pi = p0 + j;
                const unsigned b = fdiv((unsigned)pi, p.fD), d = (unsigned)pi - b * p.D;
                const unsigned m = rev ? L - 1 - l : l;
                unsigned h, w;
                if (colmajor) {
                    w = fdiv(m, p.fH);
                    h = m - w * H;
                } else {
                    h = fdiv(m, p.fW);
                    w = m - h * W;
                }
                xs[(((long long)b * 4 + kd) * p.D + d) * L + l] = sp[(j * H + h) * WP + w];
            }
        }
    }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) cross_merge_kernel(const CsmParams p) {
    pdl_wait();
    pdl_launch_dependents();
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int L = p.L, W = p.W, H = p.H, HP = p.H + 1;
    const long long p0 = (long long)blockIdx.x * p.ppc;
    const int np = (int)min((long long)p.ppc, p.planes - p0);
    T* s1 = reinterpret_cast<T*>(smem_raw);  // [ppc][W][H+1], keyed by (w, h)
    T* s3 = s1 + (size_t)p.ppc * W * HP;
    constexpr int VE = 16 / sizeof(T);
    const T* ys = static_cast<const T*>(p.in);
    T* out = static_cast<T*>(p.out);
    const unsigned n = (unsigned)(np * L);
    auto row = [&](long long pi, int kd) {
        const unsigned b = fdiv((unsigned)pi, p.fD), d = (unsigned)pi - b * p.D;
        return ys + (((long long)b * 4 + kd) * p.D + d) * L;
    };
    // stage directions 1 and 3
    for (int kd = 1; kd <= 3; kd += 2) {
        T* dst = kd == 1 ? s1 : s3;
        const bool rev = kd == 3;
        if (p.vec) {
            for (unsigned i = threadIdx.x * VE; i < n; i += kThreads * VE) {
                const unsigned j = fdiv(i, p.fL), l = i - j * L;
                Vec<T> v;
                v.v = *reinterpret_cast<const uint4*>(row(p0 + j, kd) + l);
#pragma unroll
                for (int q = 0; q < VE; ++q) {
                    const unsigned m = rev ? L - 1 - (l + q) : l + q;  // column-major position
                    const unsigned w = fdiv(m, p.fH), h = m - w * H;
                    dst[(j * W + w) * HP + h] = v.e[q];
                }
            }
        } else {
            for (unsigned i = threadIdx.x; i < n; i += kThreads) {
                const unsigned j = fdiv(i, p.fL), l = i - j * L;
                const unsigned m = rev ? L - 1 - l : l;
                const unsigned w = fdiv(m, p.fH), h = m - w * H;
                dst[(j * W + w) * HP + h] = row(p0 + j, kd)[l];
            }
        }
    }
    __syncthreads();
    // out[h, w] = (ys0[hW+w] + ys2[L-1-(hW+w)]) + (ys1[wH+h] + ys3[L-1-(wH+h)])
    if (p.vec) {
        for (unsigned i = threadIdx.x * VE; i < n; i += kThreads * VE) {
            const unsigned j = fdiv(i, p.fL), pos = i - j * L;
            const long long pi = p0 + j;
            Vec<T> v0, v2, o;
            v0.v = *reinterpret_cast<const uint4*>(row(pi, 0) + pos);
            v2.v = *reinterpret_cast<const uint4*>(row(pi, 2) + (L - VE - pos));  // reversed block
#pragma unroll
            for (int q = 0; q < VE; ++q) {
                const unsigned pq = pos + q;
                const unsigned h = fdiv(pq, p.fW), w = pq - h * W;
                const unsigned si = (j * W + w) * HP + h;
                const float a = io<T>::cvt(v0.e[q]) + io<T>::cvt(v2.e[VE - 1 - q]);
                const float c = io<T>::cvt(s1[si]) + io<T>::cvt(s3[si]);
                o.e[q] = io<T>::to(a + c);
            }
            *reinterpret_cast<uint4*>(out + pi * L + pos) = o.v;
        }
    } else {
        for (unsigned i = threadIdx.x; i < n; i += kThreads) {
            const unsigned j = fdiv(i, p.fL), pos = i - j * L;
            const long long pi = p0 + j;
            const unsigned h = fdiv(pos, p.fW), w = pos - h * W;
            const unsigned si = (j * W + w) * HP + h;
            const float a = io<T>::cvt(row(pi, 0)[pos]) + io<T>::cvt(row(pi, 2)[L - 1 - pos]);
            const float c = io<T>::cvt(s1[si]) + io<T>::cvt(s3[si]);
            out[pi * L + pos] = io<T>::to(a + c);
        }
    }
}

// ---------------------------------------------------------------- band kernels
// Maps of at least kBandMinL pixels: one CTA per band of rows of one map, so
// that even a batch-1 problem has enough CTAs.  Directions 0 and 2 of a band are
// one contiguous run of the sequence; directions 1 and 3 are W runs of one step
// per row of the band, written from (scan) or read into (merge) a [rows][W+1]
// shared tile.  The scan takes bands of kRB rows; the merge takes taller bands
// (mrb rows, chosen on the host), whose runs of directions 1 and 3 are longer
// reads (measured on GB300: 32-row fp32 bands 305 us against 337 us for 8 rows
// on the batch-128 56x56 map; 16 rows best for bf16).
constexpr int kRB = 8;
constexpr int kBandMinL = 1024;
constexpr int kBandThreads = 128;

struct BandParams {
    const void* in;
    void* out;
    int D, H, W, L;
    int nbands;  // bands per map
    int vec;     // W and H multiples of the vector width, 16-byte aligned bases
    int mrb;     // merge: rows per band (a multiple of 8)
};

template <typename T>
__global__ void __launch_bounds__(kBandThreads) cross_scan_band_kernel(const BandParams p) {
    pdl_wait();
    pdl_launch_dependents();
    extern __shared__ __align__(16) unsigned char smem_raw[];
    T* tile = reinterpret_cast<T*>(smem_raw);  // [kRB][W+1]
    constexpr int VE = 16 / sizeof(T);
    const int W = p.W, H = p.H, L = p.L, WP = p.W + 1;
    const long long plane = blockIdx.x / p.nbands;
    const int band = blockIdx.x % p.nbands;
    const int h0 = band * kRB;
    const int rb = min(kRB, H - h0);
    const int n = rb * W;
    const long long b = plane / p.D, d = plane % p.D;
    const T* src = static_cast<const T*>(p.in) + plane * L + (long long)h0 * W;
    T* xs = static_cast<T*>(p.out);
    T* row0 = xs + ((b * 4 + 0) * p.D + d) * L;
    T* row1 = xs + ((b * 4 + 1) * p.D + d) * L;
    T* row2 = xs + ((b * 4 + 2) * p.D + d) * L;
    T* row3 = xs + ((b * 4 + 3) * p.D + d) * L;
    if (p.vec) {
        for (int e = threadIdx.x * VE; e < n; e += kBandThreads * VE) {
            Vec<T> v, r;
            v.v = *reinterpret_cast<const uint4*>(src + e);
            const int j = e / W, w = e - j * W;  // a vector never crosses a row (W % VE == 0)
#pragma unroll
            for (int q = 0; q < VE; ++q) {
                tile[j * WP + w + q] = v.e[q];
                r.e[q] = v.e[VE - 1 - q];
            }
            *reinterpret_cast<uint4*>(row0 + (long long)h0 * W + e) = v.v;           // direction 0
            *reinterpret_cast<uint4*>(row2 + L - (long long)h0 * W - e - VE) = r.v;  // direction 2
        }
    } else {
        for (int e = threadIdx.x; e < n; e += kBandThreads) {
            const T v = src[e];
            const int j = e / W, w = e - j * W;
            tile[j * WP + w] = v;
            row0[(long long)h0 * W + e] = v;
            row2[L - 1 - (long long)h0 * W - e] = v;
        }
    }
    __syncthreads();
    // directions 1 and 3: for each column w, the steps w*H + h0 .. w*H + h0 + rb - 1
    if (p.vec && rb == kRB) {
        constexpr int RV = kRB / VE;  // vectors per run
        for (int i = threadIdx.x; i < W * RV; i += kBandThreads) {
            const int w = i / RV, jv = (i - w * RV) * VE;
            Vec<T> v, r;
#pragma unroll
            for (int q = 0; q < VE; ++q) {
                v.e[q] = tile[(jv + q) * WP + w];
                r.e[q] = tile[(jv + VE - 1 - q) * WP + w];
            }
            const long long pos = (long long)w * H + h0 + jv;
            *reinterpret_cast<uint4*>(row1 + pos) = v.v;
            *reinterpret_cast<uint4*>(row3 + L - pos - VE) = r.v;
        }
    } else {
        for (int e = threadIdx.x; e < n; e += kBandThreads) {
            const int w = e / rb, j = e - w * rb;
            const T v = tile[j * WP + w];
            const long long pos = (long long)w * H + h0 + j;
            row1[pos] = v;
            row3[L - 1 - pos] = v;
        }
    }
}

template <typename T>
__global__ void __launch_bounds__(kBandThreads) cross_merge_band_kernel(const BandParams p) {
    pdl_wait();
    pdl_launch_dependents();
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int W = p.W, H = p.H, L = p.L, WP = p.W + 1;
    T* s1 = reinterpret_cast<T*>(smem_raw);  // [mrb][W+1]: ys1 at pixel (h0 + j, w)
    T* s3 = s1 + p.mrb * WP;                   // [mrb][W+1]: ys3 at pixel (h0 + j, w)
    constexpr int VE = 16 / sizeof(T);
    const long long plane = blockIdx.x / p.nbands;
    const int band = blockIdx.x % p.nbands;
    const int h0 = band * p.mrb;
    const int rb = min(p.mrb, H - h0);
    const int n = rb * W;
    const long long b = plane / p.D, d = plane % p.D;
    const T* ys = static_cast<const T*>(p.in);
    const T* row0 = ys + ((b * 4 + 0) * p.D + d) * L;
    const T* row1 = ys + ((b * 4 + 1) * p.D + d) * L;
    const T* row2 = ys + ((b * 4 + 2) * p.D + d) * L;
    const T* row3 = ys + ((b * 4 + 3) * p.D + d) * L;
    T* out = static_cast<T*>(p.out) + plane * L + (long long)h0 * W;
    // stage directions 1 and 3 of the band's pixels
    if (p.vec && rb % VE == 0) {
        const int RV = rb / VE;  // vectors per run
        for (int i = threadIdx.x; i < W * RV; i += kBandThreads) {
            const int w = i / RV, jv = (i - w * RV) * VE;
            const long long pos = (long long)w * H + h0 + jv;
            Vec<T> v1, v3;
            v1.v = *reinterpret_cast<const uint4*>(row1 + pos);
            v3.v = *reinterpret_cast<const uint4*>(row3 + L - pos - VE);
#pragma unroll
            for (int q = 0; q < VE; ++q) {
                s1[(jv + q) * WP + w] = v1.e[q];
                s3[(jv + q) * WP + w] = v3.e[VE - 1 - q];
            }
        }
    } else {
        for (int e = threadIdx.x; e < n; e += kBandThreads) {
            const int w = e / rb, j = e - w * rb;
            const long long pos = (long long)w * H + h0 + j;
            s1[j * WP + w] = row1[pos];
            s3[j * WP + w] = row3[L - 1 - pos];
        }
    }
    __syncthreads();
    // out = (ys0 + ys2) + (ys1 + ys3), in this order
    if (p.vec) {
        for (int e = threadIdx.x * VE; e < n; e += kBandThreads * VE) {
            const int j = e / W, w = e - j * W;
            const long long pos = (long long)h0 * W + e;
            Vec<T> v0, v2, o;
            v0.v = *reinterpret_cast<const uint4*>(row0 + pos);
            v2.v = *reinterpret_cast<const uint4*>(row2 + L - pos - VE);
#pragma unroll
            for (int q = 0; q < VE; ++q) {
                const float a = io<T>::cvt(v0.e[q]) + io<T>::cvt(v2.e[VE - 1 - q]);
                const float c = io<T>::cvt(s1[j * WP + w + q]) + io<T>::cvt(s3[j * WP + w + q]);
                o.e[q] = io<T>::to(a + c);
            }
            *reinterpret_cast<uint4*>(out + e) = o.v;
        }
    } else {
        for (int e = threadIdx.x; e < n; e += kBandThreads) {
            const int j = e / W, w = e - j * W;
            const long long pos = (long long)h0 * W + e;
            const float a = io<T>::cvt(row0[pos]) + io<T>::cvt(row2[L - 1 - pos]);
            const float c = io<T>::cvt(s1[j * WP + w]) + io<T>::cvt(s3[j * WP + w]);
            out[e] = io<T>::to(a + c);
        }
    }
}

// Planes too large for shared memory: one thread per element, plain gathers.
template <typename T>
__global__ void cross_scan_direct(const T* x, T* xs, int D, int H, int W, long long total) {
    pdl_wait();
    pdl_launch_dependents();
    const long long L = (long long)H * W;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total; e += (long long)gridDim.x * blockDim.x) {
        const long long l = e % L, row = e / L;  // row = (b*4 + kd)*D + d
        const long long d = row % D, bk = row / D, kd = bk % 4, b = bk / 4;
        const long long m = kd >= 2 ? L - 1 - l : l;
        const long long h = (kd & 1) ? m % H : m / W;
        const long long w = (kd & 1) ? m / H : m % W;
        xs[e] = x[((b * D + d) * H + h) * W + w];
    }
}

template <typename T>
__global__ void cross_merge_direct(const T* ys, T* out, int D, int H, int W, long long total) {
    pdl_wait();
    pdl_launch_dependents();
    const long long L = (long long)H * W;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total; e += (long long)gridDim.x * blockDim.x) {
        const long long pos = e % L, pl = e / L, d = pl % D, b = pl / D;
        const long long h = pos / W, w = pos % W, p1 = w * H + h;
        const T* r = ys + (b * 4 * D + d) * L;
        const long long st = (long long)D * L;
        const float a = io<T>::cvt(r[pos]) + io<T>::cvt(r[2 * st + L - 1 - pos]);
        const float c = io<T>::cvt(r[st + p1]) + io<T>::cvt(r[3 * st + L - 1 - p1]);
        out[e] = io<T>::to(a + c);
    }
}

template <typename T>
vmb_status launch_csm(bool merge, const void* in, void* outp, int B, int D, int H, int W, cudaStream_t stream) {
    const int L = H * W;
    const long long planes = (long long)B * D;
    const size_t es = sizeof(T);
    const size_t per_plane = merge ? 2 * (size_t)W * (H + 1) * es : (size_t)H * (W + 1) * es;
    const bool small_enough = per_plane <= kMaxSmem && planes < (1ll << 31) &&
                              (long long)L * 4 < (1ll << 31);
    if (!small_enough) {
        const long long total = merge ? planes * L : planes * 4 * L;
        const int grid = (int)std::min<long long>((total + kThreads - 1) / kThreads, 152ll * 32);
        const void* fn = merge ? reinterpret_cast<const void*>(&cross_merge_direct<T>)
                               : reinterpret_cast<const void*>(&cross_scan_direct<T>);
        const T* src = static_cast<const T*>(in);
        T* dst = static_cast<T*>(outp);
        void* args[] = {&src, &dst, &D, &H, &W, const_cast<long long*>(&total)};
        return launch_kernel(fn, dim3(grid), dim3(kThreads), 0, args, stream) == cudaSuccess ? VMB_OK : VMB_ERR_CUDA;
    }
    if (L >= kBandMinL && (size_t)2 * kRB * (W + 1) * es <= kMaxSmem && planes * ((H + kRB - 1) / kRB) < (1ll << 31)) {
        BandParams bp{};
        bp.in = in;
        bp.out = outp;
        bp.D = D;
        bp.H = H;
        bp.W = W;
        bp.L = L;
        // merge bands: 32 rows (fp32) or 16 (bf16), fewer while the tiles would
        // not fit
        int mrb = es == 4 ? 32 : 16;
        while (mrb > kRB && (size_t)2 * mrb * (W + 1) * es > kMaxSmem) mrb /= 2;
        bp.mrb = mrb;
        bp.nbands = merge ? (H + mrb - 1) / mrb : (H + kRB - 1) / kRB;
        const int VE = (int)(16 / es);
        const auto a16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
        bp.vec = (W % VE == 0) && (H % VE == 0) && a16(in) && a16(outp);
        const size_t smem = merge ? 2 * (size_t)mrb * (W + 1) * es : (size_t)kRB * (W + 1) * es;
        const void* fn = merge ? reinterpret_cast<const void*>(&cross_merge_band_kernel<T>)
                               : reinterpret_cast<const void*>(&cross_scan_band_kernel<T>);
        if (smem > 48 * 1024 &&
            cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kMaxSmem) != cudaSuccess)
            return VMB_ERR_CUDA;
        void* args[] = {&bp};
        const unsigned nblk = (unsigned)(planes * bp.nbands);
        return launch_kernel(fn, dim3(nblk), dim3(kBandThreads), smem, args, stream) == cudaSuccess ? VMB_OK
                                                                                                     : VMB_ERR_CUDA;
    }
    // about 8K elements per CTA, bounded by shared memory
    int ppc = (int)std::max<long long>(1, 8192 / L);
    while (ppc > 1 && (size_t)ppc * per_plane > kMaxSmem) --ppc;
    if (ppc > planes) ppc = (int)planes;
    CsmParams p{};
    p.in = in;
    p.out = outp;
    p.D = D;
    p.H = H;
    p.W = W;
    p.L = L;
    p.planes = planes;
    p.ppc = ppc;
    const auto al16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    p.vec = ((size_t)L * es % 16 == 0) && al16(in) && al16(outp);
    p.fL = make_fastdiv((unsigned)L);
    p.fW = make_fastdiv((unsigned)W);
    p.fH = make_fastdiv((unsigned)H);
    p.fD = make_fastdiv((unsigned)D);
    const size_t smem = (size_t)ppc * per_plane;
    const void* fn = merge ? reinterpret_cast<const void*>(&cross_merge_kernel<T>)
                           : reinterpret_cast<const void*>(&cross_scan_kernel<T>);
    if (smem > 48 * 1024 && cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kMaxSmem) != cudaSuccess)
        return VMB_ERR_CUDA;
    const unsigned grid = (unsigned)((planes + ppc - 1) / ppc);
    void* args[] = {&p};
    return launch_kernel(fn, dim3(grid), dim3(kThreads), smem, args, stream) == cudaSuccess ? VMB_OK : VMB_ERR_CUDA;
}

}  // namespace

vmb_status launch_cross_scan(const void* x, void* xs, int B, int D, int H, int W, vmb_dtype dt, cudaStream_t stream) {
    return dt == VMB_BF16 ? launch_csm<__nv_bfloat16>(false, x, xs, B, D, H, W, stream)
                          : launch_csm<float>(false, x, xs, B, D, H, W, stream);
}

vmb_status launch_cross_merge(const void* ys, void* out, int B, int D, int H, int W, vmb_dtype dt, cudaStream_t stream) {
    return dt == VMB_BF16 ? launch_csm<__nv_bfloat16>(true, ys, out, B, D, H, W, stream)
                          : launch_csm<float>(true, ys, out, B, D, H, W, stream);
}

// ------------------------------------------- channel-mean path: broadcast + merge
// The channel-mean scan's output is y_k[b,d,l] = ybar_k[b,l] + Dskip[kD+d] u_k[b,d,l]
// (Eq. 9 broadcast), and every direction's u at the position it merges into is
// the map itself: u_k[b,d,p_k(h,w)] = x[b,d,h,w].  So the merged map is
//   out[b,d,h,w] = (y0 + y2) + (y1 + y3),  y_k = ybar_k[b, p_k] + Dskip[kD+d] x[b,d,h,w]
// (y_k = ybar_k[b, p_k] when the skip term is already folded into ybar), read
// from x and the four ybar rows of (b, .) without y ever being written.  The
// fp32 operations and their order are those of the broadcast and of the
// cross-merge, so fp32 results are bit-identical to the unfused path; bf16
// rounds once, at the end.  A thread owns kMP consecutive positions and keeps
// their four ybar values in registers across the CTA's channels.
namespace {
constexpr int kMMThreads = 128;
constexpr int kMP = 2;  // positions per thread
constexpr int kMMMaxDC = 64;

struct MeanMergeParams {
    const void* x;
    void* out;
    const float* ybar;   // [B, 4, L]
    const float* Dskip;  // [4 D]
    int B, D, H, W;
    int per_channel;  // 0: skip already in ybar
    int vec;          // kMP positions of a row vector-accessible (aligned rows, L % kMP == 0)
    int dc;           // channels per CTA
};

template <typename T>
__global__ void __launch_bounds__(kMMThreads) mean_merge_kernel(const MeanMergeParams p) {
    pdl_wait();
    pdl_launch_dependents();
    __shared__ float sd[4][kMMMaxDC];
    const int H = p.H, W = p.W, L = H * W;
    const int b = blockIdx.y;
    const int dbeg = blockIdx.z * p.dc, dn = min(p.dc, p.D - dbeg);
    for (int i = threadIdx.x; i < 4 * kMMMaxDC; i += kMMThreads) {
        const int kd = i / kMMMaxDC, j = i % kMMMaxDC;
        sd[kd][j] = (p.per_channel && j < dn) ? __ldg(p.Dskip + (size_t)kd * p.D + dbeg + j) : 0.0f;
    }
    const int pos0 = (blockIdx.x * kMMThreads + threadIdx.x) * kMP;
    const float* yb = p.ybar + (size_t)b * 4 * L;
    float y0[kMP], y1[kMP], y2[kMP], y3[kMP];
#pragma unroll
    for (int j = 0; j < kMP; ++j) {
        const int pos = pos0 + j;
        if (pos < L) {
            const int h = pos / W, w = pos - h * W, p1 = w * H + h;
            y0[j] = __ldg(yb + pos);
            y2[j] = __ldg(yb + 2 * (size_t)L + (L - 1 - pos));
            y1[j] = __ldg(yb + (size_t)L + p1);
            y3[j] = __ldg(yb + 3 * (size_t)L + (L - 1 - p1));
        } else {
            y0[j] = y1[j] = y2[j] = y3[j] = 0.0f;
        }
    }
    __syncthreads();
    if (pos0 >= L) return;
    const bool full = p.vec && pos0 + kMP <= L;
    const T* x = static_cast<const T*>(p.x) + ((size_t)b * p.D + dbeg) * L + pos0;
    T* out = static_cast<T*>(p.out) + ((size_t)b * p.D + dbeg) * L + pos0;
    const uint64_t ev = l2_evict_first();
    for (int dd = 0; dd < dn; ++dd, x += L, out += L) {
        float xv[kMP], o[kMP];
        if (full) {
            if constexpr (sizeof(T) == 4) {
                const float2 q = *reinterpret_cast<const float2*>(x);
                xv[0] = q.x;
                xv[1] = q.y;
            } else {
                const unsigned q = *reinterpret_cast<const unsigned*>(x);
                xv[0] = __uint_as_float(q << 16);
                xv[1] = __uint_as_float(q & 0xffff0000u);
            }
        } else {
#pragma unroll
            for (int j = 0; j < kMP; ++j) xv[j] = pos0 + j < L ? io<T>::cvt(x[j]) : 0.0f;
        }
        const float s0 = sd[0][dd], s1 = sd[1][dd], s2 = sd[2][dd], s3 = sd[3][dd];
#pragma unroll
        for (int j = 0; j < kMP; ++j) {
            const float a = fmaf(s0, xv[j], y0[j]) + fmaf(s2, xv[j], y2[j]);
            const float c = fmaf(s1, xv[j], y1[j]) + fmaf(s3, xv[j], y3[j]);
            o[j] = a + c;
        }
        if (full) {
            if constexpr (sizeof(T) == 4) {
                asm volatile("st.global.L2::cache_hint.v2.f32 [%0], {%1, %2}, %3;" ::"l"(out), "f"(o[0]), "f"(o[1]),
                             "l"(ev)
                             : "memory");
            } else {
                const unsigned q = __bfloat16_as_ushort(io<T>::to(o[0])) |
                                   ((unsigned)__bfloat16_as_ushort(io<T>::to(o[1])) << 16);
                *reinterpret_cast<unsigned*>(out) = q;
            }
        } else {
#pragma unroll
            for (int j = 0; j < kMP; ++j)
                if (pos0 + j < L) out[j] = io<T>::to(o[j]);
        }
    }
}

template <typename T>
vmb_status launch_mean_merge_t(const void* x, const float* ybar, const float* Dskip, void* out, int B, int D, int H,
                               int W, bool per_channel, cudaStream_t stream) {
    const long long L = (long long)H * W;
    const unsigned nblk = (unsigned)((L + kMMThreads * kMP - 1) / (kMMThreads * kMP));
    // channels per CTA: enough CTAs for a few waves, each amortising its ybar
    // reads over as many channels as that leaves
    const long long per_ch = (long long)nblk * B;
    long long dc = per_ch * D / (8LL * device_sm_count());
    dc = dc < 8 ? 8 : dc > kMMMaxDC ? kMMMaxDC : dc;
    if (dc > D) dc = D;
    const auto al = [](const void* q, size_t a) { return (reinterpret_cast<uintptr_t>(q) % a) == 0; };
    MeanMergeParams p{};
    p.x = x;
    p.out = out;
    p.ybar = ybar;
    p.Dskip = Dskip;
    p.B = B;
    p.D = D;
    p.H = H;
    p.W = W;
    p.per_channel = per_channel ? 1 : 0;
    p.vec = (L % kMP == 0) && al(x, kMP * sizeof(T)) && al(out, kMP * sizeof(T));
    p.dc = (int)dc;
    const dim3 grid(nblk, (unsigned)B, (unsigned)((D + dc - 1) / dc));
    if (grid.y > 65535u || grid.z > 65535u) return VMB_ERR_UNSUPPORTED;
    void* args[] = {&p};
    return launch_kernel(reinterpret_cast<const void*>(&mean_merge_kernel<T>), grid, dim3(kMMThreads), 0, args, stream) ==
                   cudaSuccess
               ? VMB_OK
               : VMB_ERR_CUDA;
}
// ------------------------------------------------------------ map transpose
// xt[b, d, w, h] = x[b, d, h, w]: the column-major order of every (b, d) plane,
// which the column-major directions of the cross-scan (1 and 3) read as
// contiguous rows.  32 x 32 tiles through shared memory (one padded column so
// the transposed reads hit distinct banks), coalesced on both sides.
constexpr int kTT = 32, kTR = 8;  // tile edge, rows per thread pass

template <typename T>
__global__ void __launch_bounds__(kTT * kTR) map_transpose_kernel(const T* x, T* xt, int H, int W, int tiles_w,
                                                                  int tiles_per_plane) {
    __shared__ T tile[kTT][kTT + 1];
    pdl_wait();
    pdl_launch_dependents();
    const long long plane = blockIdx.x / tiles_per_plane;
    const int t = blockIdx.x % tiles_per_plane;
    const int h0 = (t / tiles_w) * kTT, w0 = (t % tiles_w) * kTT;
    const T* src = x + plane * (long long)H * W;
    T* dst = xt + plane * (long long)H * W;
    const int tx = threadIdx.x % kTT, ty = threadIdx.x / kTT;
#pragma unroll
    for (int r = ty; r < kTT; r += kTR) {
        const int h = h0 + r, w = w0 + tx;
        if (h < H && w < W) tile[r][tx] = src[(long long)h * W + w];
    }
    __syncthreads();
#pragma unroll
    for (int r = ty; r < kTT; r += kTR) {
        const int w = w0 + r, h = h0 + tx;
        if (h < H && w < W) dst[(long long)w * H + h] = tile[tx][r];
    }
}

}  // namespace

vmb_status launch_map_transpose(const void* x, void* xt, int B, int D, int H, int W, vmb_dtype dt, cudaStream_t stream) {
    const int tiles_h = (H + kTT - 1) / kTT, tiles_w = (W + kTT - 1) / kTT;
    const long long grid = (long long)B * D * tiles_h * tiles_w;
    if (grid > INT32_MAX) return VMB_ERR_UNSUPPORTED;
    int tpp = tiles_h * tiles_w, tw = tiles_w;
    const void* xp = x;
    void* args[] = {&xp, &xt, &H, &W, &tw, &tpp};
    const void* fn = dt == VMB_BF16 ? reinterpret_cast<const void*>(&map_transpose_kernel<__nv_bfloat16>)
                                    : reinterpret_cast<const void*>(&map_transpose_kernel<float>);
    return launch_kernel(fn, dim3((unsigned)grid), dim3(kTT * kTR), 0, args, stream) == cudaSuccess ? VMB_OK
                                                                                                  : VMB_ERR_CUDA;
}

vmb_status launch_mean_merge(const void* x, const float* ybar, const float* Dskip, void* out, int B, int D, int H,
                             int W, bool per_channel_skip, vmb_dtype dt, cudaStream_t stream) {
    return dt == VMB_BF16
               ? launch_mean_merge_t<__nv_bfloat16>(x, ybar, Dskip, out, B, D, H, W, per_channel_skip, stream)
               : launch_mean_merge_t<float>(x, ybar, Dskip, out, B, D, H, W, per_channel_skip, stream);
}

}  // namespace vmb
