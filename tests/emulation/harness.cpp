// Runs the translated kernels on buffers of exactly the size the C ABI states
// (so AddressSanitizer sees any access outside them) and writes the outputs.
//   harness quant n k bits g kind iters sms in out : quantize, dequant, exact error
//   harness a8    n k bits g batch sms in out      : uniform quantize, int8 activations, W.A8 matmul
//   harness q4x   n k iters sms batch in out       : Q4X learner, dequant, two-matrix decode
//   harness gemv  n k bits g kind batch sms in out : quantize, then the TMA-pipelined decode
//                                                    GEMV on one matrix and on a two-entry launch
//   harness gemm  n k bits g kind m sms in out     : quantize, then the tensor-core matmul: one
//                                                    CTA per tile, split-k, split-k with PDL
//   harness q4xgemm n k iters m sms in out         : Q4X learner, then the same three matmuls
//                                                    on the Q4X weights
// `in` holds W (fp16 [n][k]) and, for a8 and q4x, x (fp16 [batch][k]).
#include <cstdio>
#include <new>
#include <string>

#include "qx_kernels.cuh"

namespace {
template <class T>
T *alloc(size_t bytes);
void put(FILE *f, const void *p, size_t b);

// qx_gemm, then qx_gemm_splitk twice on one workspace (the second with PDL):
// Y, whether the split counters are back to zero, and the plan, per run.
void three_matmuls(qx::GemmArgs base, int sms, FILE *fo) {
    uint8_t *ws = nullptr;
    for (int run = 0; run < 3; ++run) {
        const qx::GemmPlan plan = qx::plan_gemm(base.n, base.k, base.m, sms, run > 0);
        qx::GemmArgs a = base;
        __half *Y = alloc<__half>(2 * base.m * base.n);
        a.Y = Y;
        a.bn = plan.bn;
        a.splits = plan.splits;
        a.pdl = run == 2;
        if (plan.splits > 1) {
            if (ws == nullptr) {
                ws = alloc<uint8_t>(plan.ws_bytes);
                std::memset(ws, 0, plan.ws_bytes);
            }
            a.ws_cnt = reinterpret_cast<uint32_t *>(ws);
            a.ws_part = reinterpret_cast<float *>(ws + qx::kSplitCounterBytes);
        }
        qx::launch_gemm(a, sms, nullptr);
        put(fo, Y, 2 * base.m * base.n);
        uint32_t clean = 1;
        if (plan.splits > 1)
            for (size_t i = 0; i < qx::kSplitCounterBytes; ++i) clean &= ws[i] == 0;
        put(fo, &clean, 4);
        const uint32_t shape[2] = {(uint32_t)plan.bn, (uint32_t)plan.splits};
        put(fo, shape, 8);
    }
}
}  // namespace

namespace {
template <class T>
T *alloc(size_t bytes) {
    return bytes ? static_cast<T *>(::operator new(bytes, std::align_val_t(256))) : nullptr;
}
void put(FILE *f, const void *p, size_t b) {
    if (b) fwrite(p, 1, b, f);
}
bool get(FILE *f, void *p, size_t b) { return fread(p, 1, b, f) == b; }
}  // namespace

int main(int argc, char **argv) {
    if (argc < 2) return 2;
    const std::string cmd = argv[1];
    if (cmd == "q4xgemm") {  // n k iters m sms in out
        if (argc != 9) return 2;
        const int64_t n = atoll(argv[2]), k = atoll(argv[3]), m = atoll(argv[5]);
        const int iters = atoi(argv[4]), sms = atoi(argv[6]);
        FILE *fi = fopen(argv[7], "rb"), *fo = fopen(argv[8], "wb");
        if (fi == nullptr || fo == nullptr) return 2;
        const int G = (int)(k / 64), bb = (G + 3) / 4;
        __half *W = alloc<__half>(2 * n * k), *X = alloc<__half>(2 * m * k);
        if (!get(fi, W, 2 * n * k) || !get(fi, X, 2 * m * k)) return 2;
        uint32_t *status = alloc<uint32_t>(4);
        *status = 0;
        uint8_t *codes = alloc<uint8_t>(n * k / 2), *books = alloc<uint8_t>(n * bb);
        __half *scales = alloc<__half>(2 * n * G), *cbs = alloc<__half>(128);
        void *ws = alloc<uint8_t>(qx::q4x_workspace_bytes(n, k));
        qx::Q4xQuantArgs q{W, n, k, G, bb, iters, codes, scales, books, cbs, ws, status};
        qx::launch_q4x_quantize(q, sms, nullptr);
        put(fo, codes, n * k / 2);
        put(fo, scales, 2 * n * G);
        put(fo, books, n * bb);
        put(fo, cbs, 128);
        qx::GemmArgs a{};
        a.codes = codes;
        a.scales = scales;
        a.zeros = books;     // Q4X: the 2-bit book indices
        a.luts = cbs;        // Q4X: the four codebooks
        a.n = n;
        a.k = k;
        a.m = m;
        a.bits = 4;
        a.kind = 2;
        a.log2g = 6;
        a.G = G;
        a.zbytes = bb;
        a.X = X;
        a.status = status;
        a.wait_limit_ns = 60000000000ull;
        three_matmuls(a, sms, fo);
        put(fo, status, 4);
        fclose(fo);
        fclose(fi);
        return 0;
    }
    const bool q4x = cmd == "q4x";
    const int want = q4x ? 9 : (cmd == "quant" || cmd == "gemv" || cmd == "gemm") ? 11 : 10;
    if (argc != want) return 2;
    const int64_t n = atoll(argv[2]), k = atoll(argv[3]);
    FILE *fi = fopen(argv[argc - 2], "rb"), *fo = fopen(argv[argc - 1], "wb");
    if (fi == nullptr || fo == nullptr) return 2;
    __half *W = alloc<__half>(2 * n * k);
    if (!get(fi, W, 2 * n * k)) return 2;
    uint32_t *status = alloc<uint32_t>(4);
    *status = 0;
    if (q4x) {
        const int iters = atoi(argv[4]), sms = atoi(argv[5]), batch = atoi(argv[6]);
        const int G = (int)(k / 64), bb = (G + 3) / 4;
        __half *x = alloc<__half>(2 * batch * k);
        if (!get(fi, x, 2 * batch * k)) return 2;
        uint8_t *codes = alloc<uint8_t>(n * k / 2), *books = alloc<uint8_t>(n * bb);
        __half *scales = alloc<__half>(2 * n * G), *cbs = alloc<__half>(128);
        void *ws = alloc<uint8_t>(qx::q4x_workspace_bytes(n, k));
        qx::Q4xQuantArgs a{W, n, k, G, bb, iters, codes, scales, books, cbs, ws, status};
        qx::launch_q4x_quantize(a, sms, nullptr);
        qx::Q4xMat m{codes, scales, books, cbs, n, k, G, bb};
        __half *Wh = alloc<__half>(2 * n * k);
        qx::launch_q4x_dequant(m, Wh, sms, nullptr);
        float *y0 = alloc<float>(4 * batch * n), *y1 = alloc<float>(4 * batch * n);
        qx::Q4xGemvMulti g{};
        g.count = 2;
        g.batch = batch;
        g.y_f32 = 1;
        g.mat[0] = g.mat[1] = m;
        g.x[0] = g.x[1] = x;
        g.y[0] = y0;
        g.y[1] = y1;
        g.row_off[1] = n;
        g.row_off[2] = 2 * n;
        qx::launch_q4x_gemv(g, sms, nullptr);
        __half *yh = alloc<__half>(2 * batch * n);
        g.count = 1;
        g.y_f32 = 0;
        g.y[0] = yh;
        qx::launch_q4x_gemv(g, sms, nullptr);
        // the same decodes on the register-dequant kernel (kind 2; k a multiple
        // of 128): the matrix twice in fp32, then once in fp16
        float *y2 = alloc<float>(4 * batch * n), *y3 = alloc<float>(4 * batch * n);
        __half *yh2 = alloc<__half>(2 * batch * n);
        int ring = 0;
        if (k % 128 == 0) {
            for (int launch = 0; launch < 2; ++launch) {
                qx::GemvMulti r{};
                r.bits = 4;
                r.kind = 2;
                r.batch = batch;
                r.y_f32 = launch == 0;
                r.status = status;
                r.wait_limit_ns = 60000000000ull;
                r.nphase = 1;
                r.count = launch == 0 ? 2 : 1;
                r.phase_first[1] = r.count;
                for (int i = 0; i < r.count; ++i) {
                    qx::GemvMat &M = r.mat[i];
                    M.codes = codes;
                    M.scales = scales;
                    M.zeros = books;
                    M.luts = cbs;
                    M.x = x;
                    M.y = launch == 1 ? static_cast<void *>(yh2) : static_cast<void *>(i == 0 ? y2 : y3);
                    M.n = n;
                    M.k = k;
                    M.G = G;
                    M.zbytes = bb;
                    M.log2g = 6;
                }
                if (!qx::plan_gemv(r, sms)) return 3;
                qx::launch_gemv_multi(r, nullptr, false);
            }
            ring = 1;
        }
        put(fo, codes, n * k / 2);
        put(fo, scales, 2 * n * G);
        put(fo, books, n * bb);
        put(fo, cbs, 128);
        put(fo, Wh, 2 * n * k);
        put(fo, y0, 4 * batch * n);
        put(fo, y1, 4 * batch * n);
        put(fo, yh, 2 * batch * n);
        put(fo, &ring, 4);
        put(fo, y2, 4 * batch * n);
        put(fo, y3, 4 * batch * n);
        put(fo, yh2, 2 * batch * n);
    } else {
        const int bits = atoi(argv[4]), g = atoi(argv[5]);
        const bool three = cmd == "quant" || cmd == "gemv" || cmd == "gemm";  // commands that take a kind
        const int kind = three ? atoi(argv[6]) : 0;
        const int extra = atoi(argv[three ? 7 : 6]), sms = atoi(argv[three ? 8 : 7]);
        const int G = (int)(k / g), zb = (G + 1) / 2;
        const size_t cb = n * k * bits / 8, sb = kind == 0 ? 2 * n * G : 0, zbb = kind == 0 ? n * zb : 0,
                     lb = kind == 1 ? 2 * n * G * 8 : 0;
        uint8_t *codes = alloc<uint8_t>(cb), *zeros = alloc<uint8_t>(zbb);
        __half *scales = alloc<__half>(sb), *luts = alloc<__half>(lb);
        qx::QuantArgs q{W, n, k, bits, g, kind, cmd == "quant" ? extra : 25, G, zb, codes, scales, zeros, luts, status};
        qx::launch_quantize(q, sms, nullptr);
        put(fo, codes, cb);
        put(fo, scales, sb);
        put(fo, zeros, zbb);
        put(fo, luts, lb);
        if (cmd == "gemm") {
            const int64_t m = extra;
            __half *X = alloc<__half>(2 * m * k);
            if (!get(fi, X, 2 * m * k)) return 2;
            int l = 0;
            while ((1 << l) < g) ++l;
            qx::GemmArgs a{};
            a.codes = codes;
            a.scales = scales;
            a.zeros = zeros;
            a.luts = luts;
            a.n = n;
            a.k = k;
            a.m = m;
            a.bits = bits;
            a.kind = kind;
            a.log2g = l;
            a.G = G;
            a.zbytes = zb;
            a.X = X;
            a.status = status;
            a.wait_limit_ns = 60000000000ull;
            three_matmuls(a, sms, fo);
        } else if (cmd == "gemv") {
            const int batch = extra;
            __half *x = alloc<__half>(2 * batch * k);
            if (!get(fi, x, 2 * batch * k)) return 2;
            // launches: one matrix; the matrix twice (PDL); then twice more the
            // matrix twice with the CTAs balanced stage by stage (row blocks
            // split between CTAs, their partial sums in a workspace)
            float *ys[7];
            for (auto &y : ys) y = alloc<float>(4 * batch * n);
            float *part = alloc<float>(4 * 2 * qx::kMaxGemvCtas * 16 * 32);
            uint32_t *tick = alloc<uint32_t>(4 * qx::kMaxGemvCtas);
            std::memset(tick, 0, 4 * qx::kMaxGemvCtas);  // the workspace starts at zero
            int l = 0;
            while ((1 << l) < g) ++l;
            int has_split = 0;
            for (int launch = 0; launch < 4; ++launch) {
                qx::GemvMulti m{};
                m.count = launch == 0 ? 1 : 2;
                if (launch >= 2) {
                    m.split_part = part;
                    m.split_flag = tick;
                }
                m.nphase = 1;
                m.phase_first[0] = 0;
                m.phase_first[1] = m.count;
                m.bits = bits;
                m.kind = kind;
                m.batch = batch;
                m.y_f32 = 1;
                m.status = status;
                m.wait_limit_ns = 60000000000ull;  // the emulation is slow; a real stall still ends
                for (int i = 0; i < m.count; ++i) {
                    qx::GemvMat &M = m.mat[i];
                    M.codes = codes;
                    M.scales = scales;
                    M.zeros = zeros;
                    M.luts = luts;
                    M.x = x;
                    M.y = launch == 0 ? ys[0] : ys[2 * launch - 1 + i];
                    M.n = n;
                    M.k = k;
                    M.G = G;
                    M.zbytes = zb;
                    M.log2g = l;
                }
                if (!qx::plan_gemv(m, sms)) return 3;
                has_split = m.has_split;
                qx::launch_gemv_multi(m, nullptr, launch == 1);
            }
            for (auto &y : ys) put(fo, y, 4 * batch * n);
            put(fo, &has_split, 4);  // whether the balanced plan split a block
            uint32_t left = 0;  // flags not back at zero
            for (int i = 0; i < qx::kMaxGemvCtas; ++i) left += tick[i] != 0;
            put(fo, &left, 4);
        } else if (cmd == "quant") {
            __half *Wh = alloc<__half>(2 * n * k);
            qx::DequantArgs d{codes, scales, zeros, luts, n, k, bits, g, kind, G, zb, Wh};
            qx::launch_dequant(d, sms, nullptr);
            const int nb = qx::sq_error_blocks(sms);
            auto *part = alloc<unsigned long long>(16 * (size_t)nb), *tot = alloc<unsigned long long>(16);
            qx::launch_sq_error(W, Wh, n * k, part, tot, sms, nullptr);
            put(fo, Wh, 2 * n * k);
            put(fo, tot, 16);
        } else {
            const int batch = extra;
            __half *x = alloc<__half>(2 * batch * k);
            if (!get(fi, x, 2 * batch * k)) return 2;
            int8_t *qa = alloc<int8_t>(batch * k);
            float *sa = alloc<float>(4 * batch), *y = alloc<float>(4 * batch * n);
            qx::launch_quantize_act(x, batch, k, qa, sa, nullptr);
            int l = 0;
            while ((1 << l) < g) ++l;
            qx::GemvA8Args a{codes, scales, zeros, n, k, bits, G, zb, l, qa, sa, batch, y, 1};
            qx::launch_gemv_a8(a, nullptr);
            put(fo, qa, batch * k);
            put(fo, sa, 4 * batch);
            put(fo, y, 4 * batch * n);
        }
    }
    put(fo, status, 4);
    fclose(fo);
    fclose(fi);
    return 0;
}
