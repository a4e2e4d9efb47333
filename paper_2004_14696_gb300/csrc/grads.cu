// Eq. (2) for all n workers at once: g_i = (1/B) sum_{x in B_i} grad f(x, w).
//
// The n workers share w, so their minibatches are stacked into one batch of
// M = n * B rows and every forward and input-gradient GEMM is a single GEMM over
// M rows.  Only the weight gradient is per worker: G[i, W_l] = dZ_l[i]^T A_{l-1}[i]
// with K = B, a batched GEMM over the n workers that writes G directly.
//
//   gather     X = pool[idx]                                (fp32 or bf16)
//   forward    Z_l = A_{l-1} W_l^T + b_l, A_l = ReLU(Z_l)   (last layer: fp32 logits)
//   loss       per-sample cross entropy, loss_i = mean over worker i's B samples,
//              dZ_L = (softmax - onehot) / B
//   backward   G[i, W_l] = dZ_l[i]^T A_{l-1}[i],  G[i, b_l] = sum_rows dZ_l[i],
//              dZ_{l-1} = (dZ_l W_l) * 1[A_{l-1} > 0]      (ReLU'(0) = 0)
//
// GEMMs here are the SIMT path (fp32 FFMA on fp32 or bf16 operands), used for the
// fp32 workloads and for bf16 shapes the tcgen05 pass (grads_tc.cu) does not take;
// the fp32 workloads' large forward GEMMs run on the tensor cores in three tf32
// passes instead (gemm_tf32.cuh), which keeps fp32 accuracy.
#include <math.h>

#include "common.cuh"
#include "gemm_tf32.cuh"
#include "grads.cuh"

namespace dbw {

namespace tf32 {
__global__ void split_kernel(const float* __restrict__ src, int rows, int cols, int64_t lds, float* __restrict__ hi,
                             float* __restrict__ lo, int64_t ldo) {
    for (int r = blockIdx.y; r < rows; r += gridDim.y) {
        const float* s = src + (int64_t)r * lds;
        for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < cols; c += gridDim.x * blockDim.x) {
            float h, l;
            split_value(s[c], h, l);
            hi[(int64_t)r * ldo + c] = h;
            lo[(int64_t)r * ldo + c] = l;
        }
    }
}

__global__ void split4_kernel(const float* __restrict__ src, int rows, int cols, int64_t lds, float* __restrict__ hi,
                              float* __restrict__ lo, int64_t ldo) {
    const int c4 = cols / 4;
    const int64_t total = (int64_t)rows * c4;
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < total; q += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = q / c4;
        const int c = static_cast<int>(q - r * c4) * 4;
        const float4 v = *reinterpret_cast<const float4*>(src + r * lds + c);
        float4 h, l;
        split_value(v.x, h.x, l.x);
        split_value(v.y, h.y, l.y);
        split_value(v.z, h.z, l.z);
        split_value(v.w, h.w, l.w);
        *reinterpret_cast<float4*>(hi + r * ldo + c) = h;
        *reinterpret_cast<float4*>(lo + r * ldo + c) = l;
    }
}

void split(const float* src, int rows, int cols, int64_t lds, float* hi, float* lo, int64_t ldo, cudaStream_t st) {
    if (cols % 4 == 0 && lds % 4 == 0 && ldo % 4 == 0 && aligned16(src) && aligned16(hi) && aligned16(lo)) {
        const int64_t want = ((int64_t)rows * (cols / 4) + 255) / 256;
        const int blocks = static_cast<int>(want < 8 * sm_count() ? want : 8 * sm_count());
        split4_kernel<<<blocks < 1 ? 1 : blocks, 256, 0, st>>>(src, rows, cols, lds, hi, lo, ldo);
    } else {
        dim3 g((cols + 127) / 128, rows < 65535 ? rows : 65535);
        split_kernel<<<g, 128, 0, st>>>(src, rows, cols, lds, hi, lo, ldo);
    }
}

__global__ void split_t_kernel(const float* __restrict__ src, int rows, int cols, int64_t lds,
                               float* __restrict__ hiT, float* __restrict__ loT, int64_t ldt) {
    __shared__ float tile[32][33];
    const int tx = threadIdx.x, ty = threadIdx.y;
    const int c0 = blockIdx.x * 32;
    for (int64_t r0 = (int64_t)blockIdx.y * 32; r0 < rows; r0 += (int64_t)gridDim.y * 32) {
        for (int j = ty; j < 32; j += 8) {
            const int64_t r = r0 + j;
            const int c = c0 + tx;
            tile[j][tx] = (r < rows && c < cols) ? src[r * lds + c] : 0.f;
        }
        __syncthreads();
        for (int j = ty; j < 32; j += 8) {
            const int c = c0 + j;
            const int64_t r = r0 + tx;
            if (c < cols && r < rows) {
                float h, l;
                split_value(tile[tx][j], h, l);
                hiT[(int64_t)c * ldt + r] = h;
                loT[(int64_t)c * ldt + r] = l;
            }
        }
        __syncthreads();
    }
}
}  // namespace tf32

namespace {

template <typename T> __device__ __forceinline__ float to_f(T v);
template <> __device__ __forceinline__ float to_f<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

// ------------------------------------------------------------------ gather
// X[m, :] = pool[idx[m], :].  An index outside [0, S) reads row 0; the loss
// kernel poisons that worker.  With hi != nullptr (fp32 pass, first forward GEMM in
// three tf32 passes) the row's tf32 parts go to hi / lo [M, ldo] as well (ldo % 4 == 0).
template <typename T>
__global__ void gather_kernel(const float* __restrict__ pool, int64_t S, int in, const int32_t* __restrict__ idx,
                              int M, T* __restrict__ X, float* __restrict__ hi, float* __restrict__ lo, int64_t ldo) {
    for (int m = blockIdx.y; m < M; m += gridDim.y) {
        int64_t r = idx[m];
        if (r < 0 || r >= S) r = 0;
        const float* src = pool + r * in;
        T* dst = X + (int64_t)m * in;
        for (int c = (blockIdx.x * blockDim.x + threadIdx.x) * 4; c < in; c += gridDim.x * blockDim.x * 4) {
            if (c + 3 < in) {
                const float4 v = *reinterpret_cast<const float4*>(src + c);
                dst[c] = from_f<T>(v.x);
                dst[c + 1] = from_f<T>(v.y);
                dst[c + 2] = from_f<T>(v.z);
                dst[c + 3] = from_f<T>(v.w);
                if (hi) {
                    float4 h, l;
                    tf32::split_value(v.x, h.x, l.x);
                    tf32::split_value(v.y, h.y, l.y);
                    tf32::split_value(v.z, h.z, l.z);
                    tf32::split_value(v.w, h.w, l.w);
                    *reinterpret_cast<float4*>(hi + (int64_t)m * ldo + c) = h;
                    *reinterpret_cast<float4*>(lo + (int64_t)m * ldo + c) = l;
                }
            } else {
                for (int e = c; e < in; ++e) {
                    dst[e] = from_f<T>(src[e]);
                    if (hi) tf32::split_value(src[e], hi[(int64_t)m * ldo + e], lo[(int64_t)m * ldo + e]);
                }
            }
        }
    }
}

// The gather of the fp32 pass when its first layer runs in three tf32 passes: the
// gathered rows' tf32 parts row-major (hi / lo [M, ldo], when hi != nullptr) and
// transposed (hiT / loT [in, ldt], when hiT != nullptr), and X itself when X != nullptr.
// Tiles of 32 rows x 128 columns through shared memory, blocks of 32 x 8 threads: a lane
// moves 16 bytes of a row (in, ldo multiples of 4), then 4-byte pieces of the transposed
// rows, 128 contiguous bytes a warp.
__global__ void gather_parts_kernel(const float* __restrict__ pool, int64_t S, int in,
                                    const int32_t* __restrict__ idx, int M, float* __restrict__ X,
                                    float* __restrict__ hi, float* __restrict__ lo, int64_t ldo,
                                    float* __restrict__ hiT, float* __restrict__ loT, int64_t ldt) {
    __shared__ float tile[32][129];   // [row][column], padded: the transposed reads are conflict-free
    const int tx = threadIdx.x, ty = threadIdx.y;
    const int c0 = blockIdx.x * 128;
    for (int64_t m0 = (int64_t)blockIdx.y * 32; m0 < M; m0 += (int64_t)gridDim.y * 32) {
        for (int j = ty; j < 32; j += 8) {
            const int64_t m = m0 + j;
            const int c = c0 + 4 * tx;
            float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
            if (m < M && c < in) {
                int64_t r = idx[m];
                if (r < 0 || r >= S) r = 0;
                v = *reinterpret_cast<const float4*>(pool + r * in + c);
                if (X) *reinterpret_cast<float4*>(X + m * in + c) = v;
                if (hi) {
                    float4 h, l;
                    tf32::split_value(v.x, h.x, l.x);
                    tf32::split_value(v.y, h.y, l.y);
                    tf32::split_value(v.z, h.z, l.z);
                    tf32::split_value(v.w, h.w, l.w);
                    *reinterpret_cast<float4*>(hi + m * ldo + c) = h;
                    *reinterpret_cast<float4*>(lo + m * ldo + c) = l;
                }
            }
            tile[j][4 * tx] = v.x;
            tile[j][4 * tx + 1] = v.y;
            tile[j][4 * tx + 2] = v.z;
            tile[j][4 * tx + 3] = v.w;
        }
        if (hiT) {
            __syncthreads();
            for (int cc = ty; cc < 128; cc += 8) {
                const int c = c0 + cc;
                const int64_t m = m0 + tx;
                if (c < in && m < M)
                    tf32::split_value(tile[tx][cc], hiT[(int64_t)c * ldt + m], loT[(int64_t)c * ldt + m]);
            }
            __syncthreads();
        }
    }
}

// bf16 copy of the weight matrices (same flat layout as w; bias slots unused).
__global__ void cast_bf16_kernel(const float* __restrict__ w, int64_t d, __nv_bfloat16* __restrict__ wb) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < d; i += (int64_t)gridDim.x * blockDim.x)
        wb[i] = __float2bfloat16_rn(w[i]);
}

// ------------------------------------------------------------------ SIMT GEMM
// C[m, n] = sum_k A(m, k) B(k, n) over a 128 x 128 tile per CTA, 16-deep K
// slices staged in shared memory as fp32, 8 x 8 outputs per thread.  Two shared
// buffers: the next slice's global loads go to registers while the current slice
// is multiplied, then to the other buffer (every output still adds its products
// in increasing k).
//   A_K: A(m,k) = A[m*lda + k]   else A(m,k) = A[k*lda + m]
//   B_K: B(k,n) = B[n*ldb + k]   else B(k,n) = B[k*ldb + n]
// blockIdx.z is a batch index (offsets batchA / batchB).
constexpr int BM = 128, BN = 128, BK = 16;

// SPLIT (unbatched GEMMs with few output tiles): blockIdx.z is a split of K
// instead of a batch index; split z covers k in [z * kps, (z + 1) * kps) and
// writes its partial tile to part[z][M][N], which splitk_reduce_kernel sums in
// split order before the epilogue.
template <typename T, bool A_K, bool B_K, class Epi, bool SPLIT>
__global__ void __launch_bounds__(256) gemm_simt_kernel(int M, int N, int K, const T* __restrict__ A, int64_t lda,
                                                        int64_t batchA, const T* __restrict__ B, int64_t ldb,
                                                        int64_t batchB, Epi epi, int kps, float* __restrict__ part) {
    __shared__ __align__(16) float As[2][BK][BM];
    __shared__ __align__(16) float Bs[2][BK][BN];
    const int z = blockIdx.z;
    if (!SPLIT) {
        A += (int64_t)z * batchA;
        B += (int64_t)z * batchB;
    }
    const int kbeg = SPLIT ? z * kps : 0;
    const int kend = SPLIT ? (kbeg + kps < K ? kbeg + kps : K) : K;
    const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

    constexpr int LA = BM * BK / 256, LB = BN * BK / 256;   // elements per thread and slice
    float ra[LA], rb[LB];
    // global -> registers: the slice starting at k0 (element e of the tile is thread e % 256's)
    auto load = [&](int k0) {
#pragma unroll
        for (int q = 0; q < LA; ++q) {
            const int e = tid + q * 256;
            int mm, kk;
            if (A_K) { mm = e / BK; kk = e % BK; } else { kk = e / BM; mm = e % BM; }
            const int gm = m0 + mm, gk = k0 + kk;
            ra[q] = (gm < M && gk < kend) ? to_f<T>(A_K ? A[(int64_t)gm * lda + gk] : A[(int64_t)gk * lda + gm]) : 0.f;
        }
#pragma unroll
        for (int q = 0; q < LB; ++q) {
            const int e = tid + q * 256;
            int nn, kk;
            if (B_K) { nn = e / BK; kk = e % BK; } else { kk = e / BN; nn = e % BN; }
            const int gn = n0 + nn, gk = k0 + kk;
            rb[q] = (gn < N && gk < kend) ? to_f<T>(B_K ? B[(int64_t)gn * ldb + gk] : B[(int64_t)gk * ldb + gn]) : 0.f;
        }
    };
    // registers -> shared buffer ``buf``
    auto store = [&](int buf) {
#pragma unroll
        for (int q = 0; q < LA; ++q) {
            const int e = tid + q * 256;
            if (A_K) As[buf][e % BK][e / BK] = ra[q]; else As[buf][e / BM][e % BM] = ra[q];
        }
#pragma unroll
        for (int q = 0; q < LB; ++q) {
            const int e = tid + q * 256;
            if (B_K) Bs[buf][e % BK][e / BK] = rb[q]; else Bs[buf][e / BN][e % BN] = rb[q];
        }
    };
    if (kbeg < kend) {
        load(kbeg);
        store(0);
    }
    __syncthreads();
    int buf = 0;
    for (int k0 = kbeg; k0 < kend; k0 += BK) {
        const bool more = k0 + BK < kend;
        if (more) load(k0 + BK);   // in flight while this slice is multiplied
#pragma unroll
        for (int kk = 0; kk < BK; ++kk) {
            const float4 a0 = *reinterpret_cast<const float4*>(&As[buf][kk][ty * 4]);
            const float4 a1 = *reinterpret_cast<const float4*>(&As[buf][kk][64 + ty * 4]);
            const float4 b0 = *reinterpret_cast<const float4*>(&Bs[buf][kk][tx * 4]);
            const float4 b1 = *reinterpret_cast<const float4*>(&Bs[buf][kk][64 + tx * 4]);
            const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        // the other buffer was last read before the previous barrier
        if (more) store(buf ^ 1);
        __syncthreads();
        buf ^= 1;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int gm = m0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
        if (gm >= M) continue;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int gn = n0 + (j < 4 ? tx * 4 + j : 64 + tx * 4 + (j - 4));
            if (gn < N) {
                if (SPLIT)
                    part[((int64_t)z * M + gm) * N + gn] = acc[i][j];
                else
                    epi(z, gm, gn, acc[i][j]);
            }
        }
    }
}

// Sum of the splits of every output element, in split order, then the epilogue.
template <class Epi>
__global__ void splitk_reduce_kernel(int M, int N, int splits, const float* __restrict__ part, Epi epi) {
    const int64_t total = (int64_t)M * N;
    for (int64_t q = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q < total; q += (int64_t)gridDim.x * blockDim.x) {
        float v = 0.f;
        for (int sp = 0; sp < splits; ++sp) v += part[sp * total + q];
        epi(0, static_cast<int>(q / N), static_cast<int>(q % N), v);
    }
}

// forward hidden layer: A_l = ReLU(C + b)
template <typename T>
struct EpiHidden {
    const float* bias;
    T* out;
    int ldo;
    __device__ __forceinline__ void operator()(int, int m, int n, float v) const {
        v += bias[n];
        out[(int64_t)m * ldo + n] = from_f<T>(v > 0.f ? v : 0.f);
    }
    // 32 consecutive outputs of row m from column n0 (those below N): the biases are
    // loaded before any store
    __device__ __forceinline__ void row32(int m, int n0, int N, const float (&v)[32]) const {
        float b[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) b[j] = n0 + j < N ? bias[n0 + j] : 0.f;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const float x = v[j] + b[j];
            if (n0 + j < N) out[(int64_t)m * ldo + n0 + j] = from_f<T>(x > 0.f ? x : 0.f);
        }
    }
};
// forward last layer: logits = C + b (fp32)
struct EpiLogits {
    const float* bias;
    float* out;
    int ldo;
    __device__ __forceinline__ void operator()(int, int m, int n, float v) const {
        out[(int64_t)m * ldo + n] = v + bias[n];
    }
    __device__ __forceinline__ void row32(int m, int n0, int N, const float (&v)[32]) const {
        float b[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) b[j] = n0 + j < N ? bias[n0 + j] : 0.f;
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (n0 + j < N) out[(int64_t)m * ldo + n0 + j] = v[j] + b[j];
    }
};
// input gradient: dZ_{l-1} = C * 1[A_{l-1} > 0]  (a product, so a NaN-poisoned row stays NaN)
template <typename T>
struct EpiDx {
    const T* act;
    T* out;
    int ldo;
    __device__ __forceinline__ void operator()(int, int m, int n, float v) const {
        const float a = to_f<T>(act[(int64_t)m * ldo + n]);
        out[(int64_t)m * ldo + n] = from_f<T>(v * (a > 0.f ? 1.f : 0.f));
    }
};
// weight gradient of worker z: G[z, off + o * in + c]
struct EpiDW {
    float* G;
    int64_t ldG;
    int64_t off;
    int in;
    __device__ __forceinline__ void operator()(int z, int o, int c, float v) const {
        G[(int64_t)z * ldG + off + (int64_t)o * in + c] = v;
    }
};

// ------------------------------------------------------------------ loss
// One CTA per worker.  Per sample: stable log-softmax cross entropy, and
// dZ = (softmax - onehot) / B.  The worker's loss is the mean of its B sample
// losses, summed in sample order.  A sample index outside [0, S) or a label
// outside [0, C) makes the worker's loss and dZ rows NaN.
template <typename T>
__global__ void __launch_bounds__(256) softmax_xent_kernel(const float* __restrict__ logits, int C, int B,
                                                           const int32_t* __restrict__ idx, int64_t S,
                                                           const int32_t* __restrict__ labels,
                                                           float* __restrict__ sample_loss, T* __restrict__ dZ,
                                                           float* __restrict__ loss) {
    const int i = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    constexpr int kShared = 2048;   // sample losses kept in shared memory up to this B
    __shared__ float ls[kShared];
    __shared__ int bad_s;
    if (threadIdx.x == 0) bad_s = 0;
    __syncthreads();
    const float invB = 1.0f / (float)B;
    if (C <= 32) {
        // lane c holds class c; a warp's rows go in batches of 8 whose logits, sample
        // indices and labels are all loaded before the first is reduced
        for (int r0 = warp; r0 < B; r0 += 8 * nw) {
            float zv[8];
            int yv[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int r = r0 + j * nw;
                zv[j] = -INFINITY;
                yv[j] = -1;
                if (r < B) {
                    const int64_t row = (int64_t)i * B + r;
                    if (lane < C) zv[j] = logits[row * C + lane];
                    const int64_t sidx = idx[row];
                    if (sidx >= 0 && sidx < S) yv[j] = labels[sidx];
                }
            }
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int r = r0 + j * nw;
                if (r >= B) break;
                const int64_t row = (int64_t)i * B + r;
                const int y = yv[j];
                const bool bad = (y < 0 || y >= C);
                float mx = zv[j];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
                const float ex = lane < C ? expf(zv[j] - mx) : 0.f;
                float se = ex;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
                const float inv_se = 1.0f / se;
                if (lane < C) {
                    float g = ex * inv_se;
                    if (lane == y) g -= 1.0f;
                    dZ[row * C + lane] = from_f<T>(bad ? NAN : g * invB);
                }
                const float zy = __shfl_sync(0xffffffffu, zv[j], bad ? 0 : y);
                if (lane == 0) {
                    const float l = bad ? NAN : (mx + logf(se)) - zy;
                    sample_loss[row] = l;
                    if (r < kShared) ls[r] = l;
                    if (bad) bad_s = 1;
                }
            }
        }
    }
    for (int r = C <= 32 ? B : warp; r < B; r += nw) {
        const int64_t row = (int64_t)i * B + r;
        const int64_t sidx = idx[row];
        int y = -1;
        if (sidx >= 0 && sidx < S) y = labels[sidx];
        const bool bad = (y < 0 || y >= C);
        const float* z = logits + row * C;
        float mx = -INFINITY;
        for (int c = lane; c < C; c += 32) mx = fmaxf(mx, z[c]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        float se = 0.f;
        for (int c = lane; c < C; c += 32) se += expf(z[c] - mx);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
        const float inv_se = 1.0f / se;
        for (int c = lane; c < C; c += 32) {
            float g = expf(z[c] - mx) * inv_se;
            if (c == y) g -= 1.0f;
            dZ[row * C + c] = from_f<T>(bad ? NAN : g * invB);
        }
        if (lane == 0) {
            const float l = bad ? NAN : (mx + logf(se)) - z[y];
            sample_loss[row] = l;
            if (r < kShared) ls[r] = l;
            if (bad) bad_s = 1;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float acc = 0.f;
        for (int r = 0; r < B; ++r) acc += r < kShared ? ls[r] : sample_loss[(int64_t)i * B + r];
        loss[i] = bad_s ? NAN : acc * invB;
    }
}

// ------------------------------------------------------------------ bias gradient
// G[i, offb + o] = sum_{r < B} dZ[i*B + r, o], summed in row order.
template <typename T>
__global__ void bias_grad_kernel(const T* __restrict__ dZ, int out, int B, float* __restrict__ G, int64_t ldG,
                                 int64_t offb) {
    const int i = blockIdx.y;
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o >= out) return;
    const T* p = dZ + (int64_t)i * B * out + o;
    float acc = 0.f;
#pragma unroll 16
    for (int r = 0; r < B; ++r) acc += to_f<T>(p[(int64_t)r * out]);
    G[(int64_t)i * ldG + offb + o] = acc;
}

// Splits of K for an unbatched GEMM with few output tiles: enough CTAs for about
// two per SM, each split at least 4 K blocks deep; 1 = no split.
int splitk_count(int M, int N, int K, int batch) {
    if (batch != 1) return 1;
    const int tiles = ((N + BN - 1) / BN) * ((M + BM - 1) / BM);
    const int want = (2 * sm_count() + tiles - 1) / tiles;
    const int most = K / (4 * BK);
    int s = want < most ? want : most;
    return s < 1 ? 1 : s;
}

// Fills dst[e] = f(e) for e < count, each thread loading 8 values before storing any
// (so that one thread's loads are in flight together, not one per store).
template <class F>
__device__ __forceinline__ void fill_shared(float* dst, int count, F f) {
    for (int e0 = threadIdx.x; e0 < count; e0 += 8 * blockDim.x) {
        float t[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int e = e0 + u * blockDim.x;
            t[u] = e < count ? f(e) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int e = e0 + u * blockDim.x;
            if (e < count) dst[e] = t[u];
        }
    }
}

// ------------------------------------------------------------------ skinny GEMMs
// Forward GEMM with few outputs (the logits): C[m, n] = sum_k A[m, k] W[n, k] for
// N <= kSkinnyN.  W sits in shared memory; one warp per row of A, lane l taking
// k = l, l + 32, .. (coalesced) into N partial sums, which a butterfly adds across the
// warp; lane n hands output n to the epilogue.
constexpr int kSkinnyN = 16;
constexpr int kSkinnyK = 32;
constexpr size_t kSkinnySmem = 48 * 1024;

template <typename T, class Epi>
__global__ void __launch_bounds__(256) skinny_n_kernel(int M, int N, int K, const T* __restrict__ A, int64_t lda,
                                                       const T* __restrict__ W, int64_t ldw, Epi epi) {
    extern __shared__ float wsh[];   // W as [N, K] fp32
    fill_shared(wsh, N * K, [&](int e) { return to_f<T>(W[(int64_t)(e / K) * ldw + e % K]); });
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int nwarps = (gridDim.x * blockDim.x) >> 5;
    for (int m = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; m < M; m += nwarps) {
        float acc[kSkinnyN];
#pragma unroll
        for (int n = 0; n < kSkinnyN; ++n) acc[n] = 0.f;
        const T* a = A + (int64_t)m * lda;
        // 8 of the lane's elements loaded at a time, then multiplied
        for (int k0 = lane; k0 < K; k0 += 8 * 32) {
            float av[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) av[u] = k0 + 32 * u < K ? to_f<T>(a[k0 + 32 * u]) : 0.f;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int k = k0 + 32 * u;
                if (k < K) {
#pragma unroll
                    for (int n = 0; n < kSkinnyN; ++n)
                        if (n < N) acc[n] = fmaf(av[u], wsh[n * K + k], acc[n]);
                }
            }
        }
        float mine = 0.f;
#pragma unroll
        for (int n = 0; n < kSkinnyN; ++n) {
            if (n < N) {
                float v = acc[n];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                if (lane == n) mine = v;
            }
        }
        if (lane < N) epi(0, m, lane, mine);
    }
}

// The same for fp32 operands whose rows allow 16-byte loads (K, lda, ldw multiples of 4,
// A and W 16-byte aligned): no shared memory, W read through L1; lane l takes the
// 4-element groups k = 4 l, 4 l + 128, .. of its row, each group's products added in k
// order, then the butterfly.
// kTwo: two groups per pass with all their loads issued first (fewer round trips for long
// rows, at about 160 registers); else one group per pass (few registers, for K <= 256).
template <bool kTwo, class Epi>
__global__ void __launch_bounds__(128) skinny_n4_kernel(int M, int N, int K, const float* __restrict__ A, int64_t lda,
                                                        const float* __restrict__ W, int64_t ldw, Epi epi) {
    const int lane = threadIdx.x & 31;
    const int nwarps = (gridDim.x * blockDim.x) >> 5;
    for (int m = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; m < M; m += nwarps) {
        float acc[kSkinnyN];
#pragma unroll
        for (int n = 0; n < kSkinnyN; ++n) acc[n] = 0.f;
        const float* a = A + (int64_t)m * lda;
        if constexpr (kTwo) {
            // two of the lane's 4-element groups per pass, all their loads issued before the
            // products (which are added in group order, as below)
            for (int k0 = 4 * lane; k0 < K; k0 += 256) {
                const bool two = k0 + 128 < K;
                const float4 av0 = __ldg(reinterpret_cast<const float4*>(a + k0));
                const float4 av1 =
                    two ? __ldg(reinterpret_cast<const float4*>(a + k0 + 128)) : make_float4(0.f, 0.f, 0.f, 0.f);
                float4 wv0[kSkinnyN], wv1[kSkinnyN];
#pragma unroll
                for (int n = 0; n < kSkinnyN; ++n) {
                    if (n < N) {
                        wv0[n] = __ldg(reinterpret_cast<const float4*>(W + (int64_t)n * ldw + k0));
                        if (two) wv1[n] = __ldg(reinterpret_cast<const float4*>(W + (int64_t)n * ldw + k0 + 128));
                    }
                }
#pragma unroll
                for (int n = 0; n < kSkinnyN; ++n) {
                    if (n < N) {
                        float t = acc[n];
                        t = fmaf(av0.x, wv0[n].x, t);
                        t = fmaf(av0.y, wv0[n].y, t);
                        t = fmaf(av0.z, wv0[n].z, t);
                        t = fmaf(av0.w, wv0[n].w, t);
                        if (two) {
                            t = fmaf(av1.x, wv1[n].x, t);
                            t = fmaf(av1.y, wv1[n].y, t);
                            t = fmaf(av1.z, wv1[n].z, t);
                            t = fmaf(av1.w, wv1[n].w, t);
                        }
                        acc[n] = t;
                    }
                }
            }
        } else {
            for (int k = 4 * lane; k < K; k += 128) {
                const float4 av = __ldg(reinterpret_cast<const float4*>(a + k));
#pragma unroll
                for (int n = 0; n < kSkinnyN; ++n) {
                    if (n < N) {
                        const float4 wv = __ldg(reinterpret_cast<const float4*>(W + (int64_t)n * ldw + k));
                        float t = acc[n];
                        t = fmaf(av.x, wv.x, t);
                        t = fmaf(av.y, wv.y, t);
                        t = fmaf(av.z, wv.z, t);
                        t = fmaf(av.w, wv.w, t);
                        acc[n] = t;
                    }
                }
            }
        }
        float mine = 0.f;
#pragma unroll
        for (int n = 0; n < kSkinnyN; ++n) {
            if (n < N) {
                float v = acc[n];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                if (lane == n) mine = v;
            }
        }
        if (lane < N) epi(0, m, lane, mine);
    }
}

// Input-gradient GEMM with a short inner dimension (K = out <= kSkinnyK):
// dZ_{l-1}[m, c] = (sum_{o < K} dZ_l[m, o] W[o, c]) * 1[act[m, c] > 0], the products
// added in increasing o (EpiDx's arithmetic, with the 16 masks loaded before any
// store).  W and the CTA's 16 rows of dZ_l sit in shared memory; a thread per column
// computes the 16 rows' outputs.
template <typename T>
__global__ void __launch_bounds__(256) skinny_k_dx_kernel(int M, int N, int K, const T* __restrict__ dZ, int64_t ldz,
                                                          const T* __restrict__ W, int64_t ldw, EpiDx<T> epi) {
    constexpr int R = 16;                               // rows per CTA
    extern __shared__ float wsh[];                      // W as [K, N] fp32, then the CTA's dZ rows [R, K]
    float* zsh = wsh + N * K;
    fill_shared(wsh, N * K, [&](int e) { return to_f<T>(W[(int64_t)(e / N) * ldw + e % N]); });
    for (int m0 = blockIdx.y * R; m0 < M; m0 += gridDim.y * R) {
        __syncthreads();   // the previous rows' reads of zsh are done
        fill_shared(zsh, R * K, [&](int e) {
            const int m = m0 + e / K;
            return m < M ? to_f<T>(dZ[(int64_t)m * ldz + e % K]) : 0.f;
        });
        __syncthreads();
        for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < N; c += gridDim.x * blockDim.x) {
            float v[R];
#pragma unroll
            for (int j = 0; j < R; ++j) v[j] = 0.f;
            for (int o = 0; o < K; ++o) {
                const float wv = wsh[o * N + c];
#pragma unroll
                for (int j = 0; j < R; ++j) v[j] = fmaf(zsh[j * K + o], wv, v[j]);
            }
            // the ReLU masks of the R rows, all loaded before the first store
            float a[R];
#pragma unroll
            for (int j = 0; j < R; ++j) a[j] = m0 + j < M ? to_f<T>(epi.act[(int64_t)(m0 + j) * epi.ldo + c]) : 0.f;
#pragma unroll
            for (int j = 0; j < R; ++j)
                if (m0 + j < M) epi.out[(int64_t)(m0 + j) * epi.ldo + c] = from_f<T>(v[j] * (a[j] > 0.f ? 1.f : 0.f));
        }
    }
}

inline bool skinny_n_ok(int N, int K) { return N <= kSkinnyN && (size_t)N * K * 4 <= kSkinnySmem; }
inline bool skinny_k_ok(int N, int K) { return K <= kSkinnyK && ((size_t)N + 16) * K * 4 <= kSkinnySmem; }

template <typename T, bool A_K, bool B_K, class Epi>
cudaError_t run_gemm(int M, int N, int K, const T* A, int64_t lda, int64_t batchA, const T* B, int64_t ldb,
                     int64_t batchB, int batch, Epi epi, cudaStream_t st, float* split_ws = nullptr,
                     size_t split_floats = 0) {
    int splits = split_ws ? splitk_count(M, N, K, batch) : 1;
    while (splits > 1 && (size_t)splits * M * N > split_floats) --splits;
    if (splits > 1) {
        const int kps = ((K + splits - 1) / splits + BK - 1) / BK * BK;
        splits = (K + kps - 1) / kps;
        dim3 grid((N + BN - 1) / BN, (M + BM - 1) / BM, splits);
        gemm_simt_kernel<T, A_K, B_K, Epi, true><<<grid, 256, 0, st>>>(M, N, K, A, lda, 0, B, ldb, 0, epi, kps,
                                                                       split_ws);
        const int64_t total = (int64_t)M * N;
        const int blocks = static_cast<int>((total + 255) / 256 < 4 * sm_count() ? (total + 255) / 256 : 4 * sm_count());
        splitk_reduce_kernel<Epi><<<blocks, 256, 0, st>>>(M, N, splits, split_ws, epi);
        return cudaGetLastError();
    }
    dim3 grid((N + BN - 1) / BN, (M + BM - 1) / BM, batch);
    gemm_simt_kernel<T, A_K, B_K, Epi, false><<<grid, 256, 0, st>>>(M, N, K, A, lda, batchA, B, ldb, batchB, epi, K,
                                                                    nullptr);
    return cudaGetLastError();
}

template <typename T>
int worker_grads_impl(const GradsPlan& P, const float* w, const float* pool, int64_t S, const int32_t* labels,
                      const int32_t* idx, float* G, int64_t ld, float* loss, char* ws, cudaStream_t st) {
    const int L = P.L;
    const int M = P.M;
    const int B = P.B;
    T* X = reinterpret_cast<T*>(ws + P.off_x);
    float* logits = reinterpret_cast<float*>(ws + P.off_logits);
    float* sloss = reinterpret_cast<float*>(ws + P.off_sloss);
    T* dz[2] = {reinterpret_cast<T*>(ws + P.off_dz[0]), reinterpret_cast<T*>(ws + P.off_dz[1])};
    float* split_ws = P.split_floats ? reinterpret_cast<float*>(ws + P.off_split) : nullptr;
    cudaError_t e0 = cudaMemsetAsync(ws, 0, sizeof(int), st);
    if (e0 != cudaSuccess) return fail(DBW_ECUDA, "dbw_worker_grads: %s", cudaGetErrorString(e0));
    const T* wop;
    if (sizeof(T) == 2) {
        __nv_bfloat16* wb = reinterpret_cast<__nv_bfloat16*>(ws + P.off_wb);
        cast_bf16_kernel<<<4 * sm_count(), 256, 0, st>>>(w, P.d, wb);
        wop = reinterpret_cast<const T*>(wb);
    } else {
        wop = reinterpret_cast<const T*>(w);
    }
    {
        const int in = P.widths[0];
        dim3 grid((in + 1023) / 1024, M < 65535 ? M : 65535);
        if (sizeof(T) == 4 && (P.tf32[0] || P.tf32_dw[0])) {
            // the first layer's GEMMs in three tf32 passes take their X parts from the gather;
            // X itself only when one of them stays on SIMT
            const int ty = (M + 31) / 32;
            const bool need_x = !(P.tf32[0] && P.tf32_dw[0]);
            gather_parts_kernel<<<dim3((in + 127) / 128, ty < 65535 ? ty : 65535), dim3(32, 8), 0, st>>>(
                pool, S, in, idx, M, need_x ? reinterpret_cast<float*>(X) : nullptr,
                P.tf32[0] ? reinterpret_cast<float*>(ws + P.off_ahi) : nullptr,
                P.tf32[0] ? reinterpret_cast<float*>(ws + P.off_alo) : nullptr, (in + 3) / 4 * 4,
                P.tf32_dw[0] ? reinterpret_cast<float*>(ws + P.off_xthi) : nullptr,
                P.tf32_dw[0] ? reinterpret_cast<float*>(ws + P.off_xtlo) : nullptr, M);
        } else {
            gather_kernel<T><<<grid, 256, 0, st>>>(pool, S, in, idx, M, X, nullptr, nullptr, 0);
        }
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "gather launch: %s", cudaGetErrorString(e));

    // forward
    const T* Ain = X;
    for (int l = 0; l < L; ++l) {
        const int fin = P.widths[l], fout = P.widths[l + 1];
        const T* W = wop + P.offW[l];
        const float* bias = w + P.offb[l];
        const bool tc = sizeof(T) == 4 && P.tf32[l];
        float* part[4] = {nullptr, nullptr, nullptr, nullptr};
        if (tc) {
            part[0] = reinterpret_cast<float*>(ws + P.off_ahi);
            part[1] = reinterpret_cast<float*>(ws + P.off_alo);
            part[2] = reinterpret_cast<float*>(ws + P.off_whi);
            part[3] = reinterpret_cast<float*>(ws + P.off_wlo);
        }
        int* status = reinterpret_cast<int*>(ws);
        auto fwd = [&](auto epi) {
            if constexpr (sizeof(T) == 4) {
                if (tc)
                    return tf32::run(M, fout, fin, Ain, fin, W, fin, part[0], part[1], part[2], part[3], epi, status,
                                     st, /*a_parts_ready=*/l == 0);
            }
            if constexpr (sizeof(T) == 4) {
                if (fout <= kSkinnyN && fin % 4 == 0 && aligned16(Ain) && aligned16(W)) {
                    const int want = (M + 3) / 4;   // 4 rows (warps) per CTA
                    const int grid = want < 8 * sm_count() ? want : 8 * sm_count();
                    if (fin > 256)
                        skinny_n4_kernel<true><<<grid, 128, 0, st>>>(M, fout, fin, reinterpret_cast<const float*>(Ain),
                                                                     fin, reinterpret_cast<const float*>(W), fin, epi);
                    else
                        skinny_n4_kernel<false><<<grid, 128, 0, st>>>(M, fout, fin, reinterpret_cast<const float*>(Ain),
                                                                      fin, reinterpret_cast<const float*>(W), fin, epi);
                    return cudaGetLastError();
                }
            }
            if (skinny_n_ok(fout, fin)) {
                const int rows_per_cta = 8;
                const int want = (M + rows_per_cta - 1) / rows_per_cta;
                const int grid = want < 2 * sm_count() ? want : 2 * sm_count();
                skinny_n_kernel<T><<<grid, 256, (size_t)fout * fin * 4, st>>>(M, fout, fin, Ain, fin, W, fin, epi);
                return cudaGetLastError();
            }
            return run_gemm<T, true, true>(M, fout, fin, Ain, fin, 0, W, fin, 0, 1, epi, st, split_ws, P.split_floats);
        };
        if (l < L - 1) {
            T* Aout = reinterpret_cast<T*>(ws + P.off_act[l + 1]);
            e = fwd(EpiHidden<T>{bias, Aout, fout});
            Ain = Aout;
        } else {
            e = fwd(EpiLogits{bias, logits, fout});
        }
        if (e != cudaSuccess) return fail(DBW_ECUDA, "forward GEMM %d: %s", l, cudaGetErrorString(e));
    }
    const int C = P.widths[L];
    softmax_xent_kernel<T><<<P.n, 256, 0, st>>>(logits, C, B, idx, S, labels, sloss, dz[0], loss);
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "loss launch: %s", cudaGetErrorString(e));

    // backward
    int cur = 0;
    for (int l = L - 1; l >= 0; --l) {
        const int fin = P.widths[l], fout = P.widths[l + 1];
        const T* Aprev = (l == 0) ? X : reinterpret_cast<const T*>(ws + P.off_act[l]);
        const T* dZl = dz[cur];
        // per-worker weight gradient: M' = fout, N' = fin, K = B; A(o, r) = dZ[r*fout + o], B(r, c) = A[r*fin + c]
        bool dw_done = false;
        if constexpr (sizeof(T) == 4) {
            if (P.tf32_dw[l]) {
                const size_t ath = l == 0 ? P.off_xthi : P.off_athi, atl = l == 0 ? P.off_xtlo : P.off_atlo;
                e = tf32::run_dw(fout, fin, B, P.n, dZl, fout, Aprev, fin, reinterpret_cast<float*>(ws + P.off_zthi),
                                 reinterpret_cast<float*>(ws + P.off_ztlo), reinterpret_cast<float*>(ws + ath),
                                 reinterpret_cast<float*>(ws + atl), G + P.offW[l], fin, ld,
                                 reinterpret_cast<int*>(ws), st, /*act_parts_ready=*/l == 0);
                dw_done = true;
            }
        }
        if (!dw_done)
            e = run_gemm<T, false, false>(fout, fin, B, dZl, fout, (int64_t)B * fout, Aprev, fin, (int64_t)B * fin,
                                          P.n, EpiDW{G, ld, P.offW[l], fin}, st);
        if (e != cudaSuccess) return fail(DBW_ECUDA, "dW GEMM %d: %s", l, cudaGetErrorString(e));
        bias_grad_kernel<T><<<dim3((fout + 127) / 128, P.n), 128, 0, st>>>(dZl, fout, B, G, ld, P.offb[l]);
        e = cudaGetLastError();
        if (e != cudaSuccess) return fail(DBW_ECUDA, "bias grad %d: %s", l, cudaGetErrorString(e));
        if (l > 0) {
            // dZ_{l-1}[m, c] = sum_o dZ_l[m, o] W_l[o, c]: A(m, o) = dZ[m*fout + o], B(o, c) = W[o*fin + c]
            T* dnext = dz[cur ^ 1];
            if (skinny_k_ok(fin, fout)) {
                const int ry = (M + 15) / 16;
                dim3 grid((fin + 255) / 256, ry < 65535 ? ry : 65535);
                skinny_k_dx_kernel<T><<<grid, 256, ((size_t)fin + 16) * fout * 4, st>>>(M, fin, fout, dZl, fout,
                                                                                  wop + P.offW[l], fin,
                                                                                  EpiDx<T>{Aprev, dnext, fin});
                e = cudaGetLastError();
            } else {
                e = run_gemm<T, true, false>(M, fin, fout, dZl, fout, 0, wop + P.offW[l], fin, 0, 1,
                                             EpiDx<T>{Aprev, dnext, fin}, st, split_ws, P.split_floats);
            }
            if (e != cudaSuccess) return fail(DBW_ECUDA, "dX GEMM %d: %s", l, cudaGetErrorString(e));
            cur ^= 1;
        }
    }
    return DBW_OK;
}

}  // namespace

bool make_grads_plan(int L, const int32_t* widths, int n, int B, int prec, GradsPlan* P) {
    if (L < 1 || L > DBW_LMAX || n < 1 || n > DBW_NMAX || B < 1) return false;
    if (prec != DBW_PREC_FP32 && prec != DBW_PREC_BF16) return false;
    P->L = L;
    P->n = n;
    P->B = B;
    P->prec = prec;
    const int64_t M = (int64_t)n * B;
    if (M > (1LL << 30)) return false;
    P->M = (int)M;
    int maxw = 0;
    int64_t off = 0;
    for (int l = 0; l <= L; ++l) {
        if (widths[l] < 1 || widths[l] > (1 << 20)) return false;
        P->widths[l] = widths[l];
        if (widths[l] > maxw) maxw = widths[l];
    }
    if (widths[L] < 2) return false;
    for (int l = 0; l < L; ++l) {
        P->offW[l] = off;
        off += (int64_t)widths[l + 1] * widths[l];
        P->offb[l] = off;
        off += widths[l + 1];
    }
    P->d = off;
    const size_t es = prec == DBW_PREC_BF16 ? 2 : 4;
    size_t cur = 0;
    auto take = [&](size_t bytes) {
        const size_t at = cur;
        cur += (bytes + 255) / 256 * 256;
        return at;
    };
    take(256);   // status word (int32 at offset 0), as in the tcgen05 plan
    P->off_x = take((size_t)M * widths[0] * es);
    P->off_act[0] = P->off_x;
    for (int l = 1; l < L; ++l) P->off_act[l] = take((size_t)M * widths[l] * es);
    P->off_logits = take((size_t)M * widths[L] * 4);
    P->off_sloss = take((size_t)M * 4);
    P->off_dz[0] = take((size_t)M * maxw * es);
    P->off_dz[1] = take((size_t)M * maxw * es);
    P->off_wb = prec == DBW_PREC_BF16 ? take((size_t)P->d * 2) : 0;
    // split-K scratch of the forward and input-gradient GEMMs (the largest splits x M x N)
    size_t split = 0;
    for (int l = 0; l < L; ++l) {
        const int fin = widths[l], fout = widths[l + 1];
        const size_t f = (size_t)splitk_count(P->M, fout, fin, 1) * P->M * fout;
        const size_t x = l > 0 ? (size_t)splitk_count(P->M, fin, fout, 1) * P->M * fin : 0;
        split = f > split ? f : split;
        split = x > split ? x : split;
    }
    P->split_floats = split;
    P->off_split = split ? take(split * 4) : 0;
    // forward GEMMs with at least 2^27 multiply-adds and 32 outputs run in three tf32 passes
    size_t a_parts = 0, w_parts = 0;
    for (int l = 0; l < L; ++l) {
        const int fin = widths[l], fout = widths[l + 1];
        P->tf32[l] = prec == DBW_PREC_FP32 && fout >= 32 && (int64_t)P->M * fout * fin >= (int64_t(1) << 27);
        if (!P->tf32[l]) continue;
        const size_t ld4 = (size_t)(fin + 3) / 4 * 4;
        a_parts = (size_t)P->M * ld4 > a_parts ? (size_t)P->M * ld4 : a_parts;
        w_parts = (size_t)fout * ld4 > w_parts ? (size_t)fout * ld4 : w_parts;
    }
    P->off_ahi = a_parts ? take(a_parts * 4) : 0;
    P->off_alo = a_parts ? take(a_parts * 4) : 0;
    P->off_whi = w_parts ? take(w_parts * 4) : 0;
    P->off_wlo = w_parts ? take(w_parts * 4) : 0;
    // weight gradients with at least 2^25 multiply-adds run in three tf32 passes when each
    // worker's samples are whole 32-deep K blocks (at most 256) and the G rows of the layer
    // take 16-byte stores
    size_t zt = 0, at = 0;
    for (int l = 0; l < L; ++l) {
        const int fin = widths[l], fout = widths[l + 1];
        P->tf32_dw[l] = prec == DBW_PREC_FP32 && B % 32 == 0 && B <= tf32::dw::kMaxK && fin % 4 == 0 &&
                        P->offW[l] % 4 == 0 && fout >= 32 && (int64_t)n * fout * fin * B >= (int64_t(1) << 25);
        if (!P->tf32_dw[l]) continue;
        zt = (size_t)fout * P->M > zt ? (size_t)fout * P->M : zt;
        if (l > 0) at = (size_t)fin * P->M > at ? (size_t)fin * P->M : at;
    }
    P->off_zthi = zt ? take(zt * 4) : 0;
    P->off_ztlo = zt ? take(zt * 4) : 0;
    P->off_athi = at ? take(at * 4) : 0;
    P->off_atlo = at ? take(at * 4) : 0;
    const size_t xt = P->tf32_dw[0] ? (size_t)widths[0] * P->M : 0;
    P->off_xthi = xt ? take(xt * 4) : 0;
    P->off_xtlo = xt ? take(xt * 4) : 0;
    P->ws_bytes = cur;
    return true;
}

int grads_activations(int L, const int32_t* widths, int n, int B, int prec, int layer, size_t* offset, int64_t* ld,
                      int* elem_bytes) {
    if (layer < 1 || layer >= L) return fail(DBW_EINVAL, "dbw_worker_grads_activations: layer must be in [1, L-1]");
    if (tc_eligible(prec, B)) {
        TcPlan T;
        if (!make_tc_plan(L, widths, n, B, &T)) return fail(DBW_EINVAL, "dbw_worker_grads_activations: invalid shape");
        *offset = T.off_act[layer];
        *ld = T.ldact[layer];
        *elem_bytes = 2;
        return DBW_OK;
    }
    GradsPlan P;
    if (!make_grads_plan(L, widths, n, B, prec, &P)) return fail(DBW_EINVAL, "dbw_worker_grads_activations: invalid shape");
    *offset = P.off_act[layer];
    *ld = widths[layer];
    *elem_bytes = prec == DBW_PREC_BF16 ? 2 : 4;
    return DBW_OK;
}

size_t grads_workspace_bytes(int L, const int32_t* widths, int n, int B, int prec) {
    if (tc_eligible(prec, B)) {
        TcPlan T;
        if (!make_tc_plan(L, widths, n, B, &T)) return 0;
        return T.ws_bytes;
    }
    GradsPlan P;
    if (!make_grads_plan(L, widths, n, B, prec, &P)) return 0;
    return P.ws_bytes;
}

int launch_worker_grads(int L, const int32_t* widths, int prec, const float* w, int64_t d, const float* pool,
                        int64_t S, const int32_t* labels, const int32_t* idx, int n, int B, float* G, int64_t ld,
                        float* loss, void* ws, size_t ws_bytes, cudaStream_t st) {
    GradsPlan P;
    if (!make_grads_plan(L, widths, n, B, prec, &P)) return fail(DBW_EINVAL, "dbw_worker_grads: invalid model shape");
    if (P.d != d) return fail(DBW_EINVAL, "dbw_worker_grads: d = %lld but the widths give %lld", (long long)d,
                              (long long)P.d);
    if (!tc_eligible(prec, B) && ws_bytes < P.ws_bytes)
        return fail(DBW_EINVAL, "dbw_worker_grads: workspace %zu bytes < %zu needed", ws_bytes, P.ws_bytes);
    if (tc_eligible(prec, B)) {
        TcPlan T;
        if (!make_tc_plan(L, widths, n, B, &T)) return fail(DBW_EINVAL, "dbw_worker_grads: invalid model shape");
        if (ws_bytes < T.ws_bytes)
            return fail(DBW_EINVAL, "dbw_worker_grads: workspace %zu bytes < %zu needed", ws_bytes, T.ws_bytes);
        return worker_grads_tc(T, w, pool, S, labels, idx, G, ld, loss, static_cast<char*>(ws), st);
    }
    if (prec == DBW_PREC_BF16)
        return worker_grads_impl<__nv_bfloat16>(P, w, pool, S, labels, idx, G, ld, loss, static_cast<char*>(ws), st);
    return worker_grads_impl<float>(P, w, pool, S, labels, idx, G, ld, loss, static_cast<char*>(ws), st);
}

}  // namespace dbw
