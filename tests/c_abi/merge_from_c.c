/* A whole merge through the C ABI from plain C (C11 + the CUDA runtime, no Python):
 * two replicas ingest their deliveries, one replica unions the other in, and the
 * union is rendered. Used by tests/test_c_abi.py, which writes the inputs and checks
 * the outputs against the CPU oracle.
 *
 *   merge_from_c L H d OUT_K OUT_V  R T K_PATH V_PATH  [R T K_PATH V_PATH ...]
 *
 * Each delivery names its replica R (0 or 1), its length T and two files of raw bf16
 * bits [L][H][T][d]. The program prints one line per delivery ("delivery <i> <id hex>
 * <absorbed>"), then "size <n>", "seq_len <n>" and "order <id hex>..." for the rendered
 * union, and writes the rendered K and V ([L][H][seq_len][d] bf16 bits) to OUT_K and
 * OUT_V. Exit status 0 on success. */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>

#include <cuda_runtime.h>

#include "cm.h"

#define MAX_DELIVERIES 16

static int fail_cm(const char *what, cm_status st) {
    fprintf(stderr, "%s: %s (%s)\n", what, cm_status_string(st), cm_last_error_message());
    return 1;
}

static int fail_cuda(const char *what, cudaError_t e) {
    fprintf(stderr, "%s: %s\n", what, cudaGetErrorString(e));
    return 1;
}

static void *read_file(const char *path, size_t bytes) {
    FILE *f = fopen(path, "rb");
    if (!f) return NULL;
    void *buf = malloc(bytes ? bytes : 1);
    if (buf && fread(buf, 1, bytes, f) != bytes) {
        free(buf);
        buf = NULL;
    }
    fclose(f);
    return buf;
}

static int write_file(const char *path, const void *buf, size_t bytes) {
    FILE *f = fopen(path, "wb");
    if (!f) return 1;
    const int bad = fwrite(buf, 1, bytes, f) != bytes;
    return fclose(f) != 0 || bad;
}

static void print_id(const cm_id *id) {
    for (int i = 0; i < 16; ++i) printf("%02x", id->b[i]);
}

int main(int argc, char **argv) {
    if (argc < 10 || (argc - 6) % 4 != 0) {
        fprintf(stderr, "usage: %s L H d OUT_K OUT_V (R T K_PATH V_PATH)...\n", argv[0]);
        return 2;
    }
    const int32_t L = atoi(argv[1]), H = atoi(argv[2]), d = atoi(argv[3]);
    const char *out_k_path = argv[4], *out_v_path = argv[5];
    const int n = (argc - 6) / 4;
    if (n > MAX_DELIVERIES) return 2;

    cm_context *ctx = NULL;
    cm_set *replica[2] = {NULL, NULL};
    cm_status st = cm_context_create(0, 1.0e6, -1, 0, &ctx);
    if (st != CM_OK) return fail_cm("cm_context_create", st);
    for (int r = 0; r < 2; ++r)
        if ((st = cm_set_create(ctx, &replica[r])) != CM_OK) return fail_cm("cm_set_create", st);

    void *dev_k[MAX_DELIVERIES] = {0}, *dev_v[MAX_DELIVERIES] = {0};
    for (int i = 0; i < n; ++i) {
        const int r = atoi(argv[6 + 4 * i]);
        const int32_t T = atoi(argv[7 + 4 * i]);
        if (r < 0 || r > 1 || T < 1) return 2;
        const size_t bytes = (size_t)L * H * T * d * 2;
        void *hk = read_file(argv[8 + 4 * i], bytes), *hv = read_file(argv[9 + 4 * i], bytes);
        if (!hk || !hv) {
            fprintf(stderr, "cannot read delivery %d\n", i);
            return 1;
        }
        cudaError_t e = cudaMalloc(&dev_k[i], bytes);
        if (e == cudaSuccess) e = cudaMalloc(&dev_v[i], bytes);
        if (e == cudaSuccess) e = cudaMemcpy(dev_k[i], hk, bytes, cudaMemcpyHostToDevice);
        if (e == cudaSuccess) e = cudaMemcpy(dev_v[i], hv, bytes, cudaMemcpyHostToDevice);
        free(hk);
        free(hv);
        if (e != cudaSuccess) return fail_cuda("fragment upload", e);
        /* Ingest(S, C) of Algorithm 2 into the delivery's replica */
        cm_fragment frag = {L, H, T, d, dev_k[i], dev_v[i]};
        cm_id id;
        int32_t absorbed = 0;
        if ((st = cm_ingest(replica[r], &frag, NULL, &id, &absorbed)) != CM_OK)
            return fail_cm("cm_ingest", st);
        printf("delivery %d ", i);
        print_id(&id);
        printf(" %d\n", absorbed);
    }

    /* Merge of Algorithm 2: replica 0 := replica 0 u replica 1 */
    if ((st = cm_union(replica[0], replica[1])) != CM_OK) return fail_cm("cm_union", st);
    int64_t size = 0, total = 0;
    cm_set_size(replica[0], &size);
    cm_set_seq_len(replica[0], &total);

    /* Render of Algorithm 2 (CanonicalMerge) into [L][H][total][d] */
    const size_t out_bytes = (size_t)L * H * (size_t)total * d * 2;
    void *k_out = NULL, *v_out = NULL;
    cudaError_t e = cudaMalloc(&k_out, out_bytes ? out_bytes : 16);
    if (e == cudaSuccess) e = cudaMalloc(&v_out, out_bytes ? out_bytes : 16);
    if (e != cudaSuccess) return fail_cuda("output allocation", e);
    cm_id order[MAX_DELIVERIES];
    int64_t seq_len = -1;
    if ((st = cm_render(replica[0], k_out, v_out, total, NULL, &seq_len, order)) != CM_OK)
        return fail_cm("cm_render", st);
    if ((st = cm_context_check(ctx, NULL)) != CM_OK) return fail_cm("cm_context_check", st);
    void *hk = malloc(out_bytes ? out_bytes : 1), *hv = malloc(out_bytes ? out_bytes : 1);
    if (!hk || !hv) return 1;
    e = cudaMemcpy(hk, k_out, out_bytes, cudaMemcpyDeviceToHost);
    if (e == cudaSuccess) e = cudaMemcpy(hv, v_out, out_bytes, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return fail_cuda("output download", e);
    if (write_file(out_k_path, hk, out_bytes) || write_file(out_v_path, hv, out_bytes)) {
        fprintf(stderr, "cannot write the outputs\n");
        return 1;
    }
    printf("size %lld\nseq_len %lld\norder", (long long)size, (long long)seq_len);
    for (int64_t i = 0; i < size; ++i) {
        printf(" ");
        print_id(&order[i]);
    }
    printf("\n");

    free(hk);
    free(hv);
    cudaFree(k_out);
    cudaFree(v_out);
    for (int r = 0; r < 2; ++r) cm_set_destroy(replica[r]);
    for (int i = 0; i < n; ++i) {
        cudaFree(dev_k[i]);
        cudaFree(dev_v[i]);
    }
    cm_context_destroy(ctx);
    return 0;
}
